"""Helpers for the GPU parity tests: build caches, copy a unit to the host as
bf16 bit patterns, and compare one eviction event of the CUDA path with the
fp64 oracle fed the same pre-eviction bytes (step-locked).

Acceptance (per event, per unit):
* scores: |s_gpu - s_ora| <= 1e-5 s_ora + atol, where atol is the fp32
  rounding floor of the GPU's arithmetic: 2e-6 (|v_j| + |mean|) for L2 (the
  squared deviation is a sum of d fp32 terms of size up to (|v_j|+|mean|)^2),
  1e-6 for Dir (a difference of unit vectors) and 0 for Norm;
* kept sets: identical, except for tokens whose oracle score lies within
  1e-5 s_(N) of the N-th largest oracle score s_(N) (near ties that fp32
  rounding may order either way);
* compacted K and V: bit-identical to the pre-eviction rows at the GPU's kept
  indices, which are strictly ascending; the length becomes N exactly.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2609_23314_gb300 as vd

RTOL = 1e-5


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def new_cache(n_seq, n_layer, n_kv_head, capacity, d, device="cuda"):
    return vd.Cache.empty(n_seq, n_layer, n_kv_head, capacity, d, device=device)


def units_view(t: torch.Tensor) -> torch.Tensor:
    """[n_seq, L, H, cap, d] -> [U, cap, d] view."""
    return t.view(-1, t.shape[-2], t.shape[-1])


def score_tolerance(var, s_ora, v_rows, mu):
    if var == oracle.L2:
        vn = np.linalg.norm(oracle.bits_to_float(v_rows), axis=1)
        return RTOL * s_ora + 2e-6 * (vn + np.linalg.norm(mu))
    if var == oracle.DIR:
        return RTOL * s_ora + 1e-6
    return RTOL * s_ora


def check_scores(orc, var, pre_v, s_gpu):
    s_ora = orc.scores(pre_v, var)
    mu = orc.mean(pre_v)
    tol = score_tolerance(var, s_ora, pre_v, mu)
    err = np.abs(s_gpu.astype(np.float64) - s_ora)
    bad = np.flatnonzero(err > tol)
    assert bad.size == 0, (f"{bad.size} scores out of tolerance; worst rel "
                           f"{np.max(err / np.maximum(s_ora, 1e-30)):.3e} at {bad[:5]}")
    return s_ora


def near_tie_band(s_ora, N):
    s_n = np.sort(s_ora)[::-1][N - 1]
    return np.abs(s_ora - s_n) <= RTOL * s_n + 1e-12


def check_event(orc, var, pre_k, pre_v, post_k, post_v, n, N, kept_gpu=None, scores_gpu=None,
                new_len=None):
    """One unit, one event.  pre_*: uint16 [>= n, d] before the call; post_*:
    uint16 [>= N, d] after it; kept_gpu: int32 [N_stride] or None."""
    pre_k, pre_v = pre_k[:n], pre_v[:n]
    if n <= N:
        if new_len is not None:
            assert new_len == n
        assert np.array_equal(post_k[:n], pre_k) and np.array_equal(post_v[:n], pre_v)
        if kept_gpu is not None:
            assert np.array_equal(kept_gpu[:n], np.arange(n)) and np.all(kept_gpu[n:] == -1)
        return None
    if new_len is not None:
        assert new_len == N
    s_ora = orc.scores(pre_v, var)
    if scores_gpu is not None:
        check_scores(orc, var, pre_v, scores_gpu[:n])
    kept_ora = orc.select_top_n(s_ora, N)
    if kept_gpu is None:
        # recover the GPU's kept list from the moved V rows is ambiguous with
        # duplicates: compare bytes against the oracle gather where the sets agree
        k2, v2, _, _ = orc.evict_unit(pre_k, pre_v, N, var)
        same = np.array_equal(post_v[:N], v2) and np.array_equal(post_k[:N], k2)
        if not same:
            band = near_tie_band(s_ora, N)
            assert band.sum() > 1, "compacted rows differ from the oracle outside any near tie"
        return kept_ora
    kg = np.asarray(kept_gpu[:N], dtype=np.int64)
    assert np.all(np.diff(kg) > 0) and kg[0] >= 0 and kg[-1] < n, "kept list not ascending/in range"
    diff = np.setxor1d(kg, kept_ora)
    if diff.size:
        band = near_tie_band(s_ora, N)
        assert np.all(band[diff]), f"kept sets differ outside the near-tie band at {diff[:8]}"
    assert np.array_equal(post_k[:N], pre_k[kg]), "K rows not gathered bit-exactly"
    assert np.array_equal(post_v[:N], pre_v[kg]), "V rows not gathered bit-exactly"
    return kept_ora
