"""Helpers for the GPU parity tests: build caches, copy a unit to the host as
bf16 bit patterns, and compare one eviction event of the CUDA path with the
fp64 oracle fed the same pre-eviction bytes (step-locked).

Acceptance (per event, per unit):
* scores: |s_gpu - s_ora| <= 1e-5 s_ora + atol (the relative tolerance the
  method's definition is checked at), where atol only covers the accuracy of
  the mean itself (~1e-11 of the data's scale) and, for Dir, a 1.8e-12
  floor (score_tolerance derives both);
* kept sets: identical, except for tokens whose oracle score lies within
  1e-5 s_(N) of the N-th largest oracle score s_(N) (near ties that fp32
  rounding may order either way);
* compacted K and V: bit-identical to the pre-eviction rows at the GPU's kept
  indices, which are strictly ascending; the length becomes N exactly.

Every score comparison also records the worst relative error it saw, per test
and rule (``record_error``); the session prints the table at the end.
"""
from __future__ import annotations

import os

import numpy as np
import torch

import oracle
import paper_2609_23314_gb300 as vd

RTOL = 1e-5
# Relative accuracy of the kernel's mean (double-float column sums, fp64
# division, an fp32 part plus an fp32 remainder) with respect to the mean of
# |v|: the same 1e-12 the running-sum checks hold the sums to.
MEAN_RTOL = 1e-12
VAR_NAMES = {oracle.L2: "l2", oracle.DIR: "dir", oracle.NORM: "norm"}
# Dir: the second-order effect of a 32-ulp error in |v| / |mean| (below)
DIR_RADIAL_FLOOR = 0.5 * (32 * 2.0 ** -24) ** 2

# (test, rule) -> [worst |ds| / s over scores > 1e-6, worst |ds| / tolerance, count]
WORST: dict = {}
# workload -> summary of a free-running trajectory (test_gpu_trajectory.py)
TRAJECTORIES: dict = {}


def record_error(var, s_gpu, s_ora, tag: str = "", tol=None):
    """Tracks, for the session summary, the worst relative score error (over
    scores above 1e-6, where the relative tolerance is the one that binds)
    and the worst error as a fraction of the tolerance (1.0 would fail)."""
    test = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0].split("::")[-1]
    key = (test, VAR_NAMES.get(var, str(var)) + tag)
    s_ora = np.asarray(s_ora, np.float64)
    err = np.abs(np.asarray(s_gpu, np.float64) - s_ora)
    big = s_ora > 1e-6
    rel = float(np.max(err[big] / s_ora[big])) if np.any(big) else 0.0
    frac = 0.0
    if tol is not None:
        t = np.broadcast_to(np.asarray(tol, np.float64), s_ora.shape)
        ok = t > 0
        frac = float(np.max(err[ok] / t[ok])) if np.any(ok) else 0.0
    w = WORST.setdefault(key, [0.0, 0.0, 0])
    w[0] = max(w[0], rel)
    w[1] = max(w[1], frac)
    w[2] += int(s_ora.size)


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> numpy uint16 bit patterns (host copy)."""
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def new_cache(n_seq, n_layer, n_kv_head, capacity, d, device="cuda"):
    return vd.Cache.empty(n_seq, n_layer, n_kv_head, capacity, d, device=device)


def units_view(t: torch.Tensor) -> torch.Tensor:
    """[n_seq, L, H, cap, d] -> [U, cap, d] view."""
    return t.view(-1, t.shape[-2], t.shape[-1])


def score_tolerance(var, s_ora, v_rows, mu):
    """Allowed |s_gpu - s_ora| per row: RTOL * s_ora plus an absolute term
    that covers only the error of the kernel's mean.

    Every rounding the kernel does after the mean is relative to the score
    itself: the mean enters as an fp32 part plus its fp32 remainder, so
    L2's deviation (v - hi) - lo is rounded relative to v - mean; the squares
    and the d-term sums (fp32, at most ~12 levels deep) and the square root
    add a few 2^-24 relative; Dir's w = v - (|v|/|m|) m is one fused
    multiply-add per element against the same two-part mean, its radial error
    (from |v| and |m|) changes the score relatively, and the final division
    by |v|^2 is one more rounding.  Worst case well under 1e-5 (about 50
    ulp for Dir, 10 for L2; observed far less).

    What is not relative: the mean's own error dm, |dm| <= MEAN_RTOL * mean|v|
    per coordinate.  It moves an L2 score by at most |dm| and a Dir score by
    at most sqrt(2 s) |dm| / |m|.  And for Dir, the second-order part of the
    radial error: with |v|/|m| off by a relative delta, |w|^2 gains
    |v|^2 delta^2 on top of the first-order (relative) change, so a row
    parallel to the mean (s = 0) scores delta^2 / 2.  delta is at most ~32
    ulp (|v| and |m| from fp32 sums, two square roots, a product), a floor of
    0.5 (32 * 2^-24)^2 = 1.8e-12.  Norm reads no mean: purely relative."""
    s_ora = np.asarray(s_ora, np.float64)
    if var == oracle.NORM:
        return RTOL * s_ora
    vals = oracle.bits_to_float(v_rows)
    dm = MEAN_RTOL * np.linalg.norm(np.abs(vals).mean(axis=0))
    if var == oracle.L2:
        return RTOL * s_ora + dm
    mn = np.linalg.norm(mu)
    first = np.sqrt(2.0 * np.maximum(s_ora, 0.0)) * dm / mn if mn > 0 else 0.0
    return RTOL * s_ora + first + DIR_RADIAL_FLOOR


def weighted_tolerance(var, s_weighted, base, v_rows, mu, f):
    """The attention-weighted score a/(1 - a) * s (App. A): the factor and
    the product add three fp32 roundings (relative); the mean's absolute
    term scales with the factor."""
    s_weighted = np.asarray(s_weighted, np.float64)
    return RTOL * np.abs(s_weighted) + (score_tolerance(var, base, v_rows, mu)
                                        - RTOL * np.asarray(base, np.float64)) * f


def check_scores(orc, var, pre_v, s_gpu):
    s_ora = orc.scores(pre_v, var)
    mu = orc.mean(pre_v)
    tol = score_tolerance(var, s_ora, pre_v, mu)
    err = np.abs(s_gpu.astype(np.float64) - s_ora)
    record_error(var, s_gpu, s_ora, tol=tol)
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
