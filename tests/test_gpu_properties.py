"""Properties of the CUDA path that the mathematics fixes, checked on the GPU
without the oracle: positive homogeneity of the scores (Sec. 3.2: L2 and Norm
scale with the values, Dir does not), permutation equivariance of the kept
set (Eq. eviction ranks tokens, not slots), translation invariance of the
L2 score (a constant shift of every value moves the mean with it), and the
L2 score as the uniform-attention disturbance of Sec. 3.3.  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import bits, near_tie_band, new_cache, record_error, score_tolerance, units_view

pytestmark = pytest.mark.gpu
VARIANTS = [vd.VD_SCORE_L2, vd.VD_SCORE_DIR, vd.VD_SCORE_NORM]
VAR_IDS = ["l2", "dir", "norm"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def filled(n, d, seed, units=4, cap=None):
    cache = new_cache(1, 1, units, cap or n, d)
    st = wl.TokenStream("gauss_outlier", units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap or n)
    cache.len.fill_(n)
    return cache


def scores_of(cache, var):
    out = torch.full(cache.unit_shape() + (cache.capacity,), float("nan"), device="cuda")
    vd.vd_score(cache, var, out)
    assert vd.vd_get_device_status() == 0
    return out.view(cache.units, -1)


def evict(cache, N, var):
    kept = torch.full(cache.unit_shape() + (N,), -1, dtype=torch.int32, device="cuda")
    scores = torch.full(cache.unit_shape() + (cache.capacity,), float("nan"), device="cuda")
    vd.vd_evict_block(cache, N, None, 0, var, vd.VD_MU_RECOMPUTE, None, kept, scores)
    assert vd.vd_get_device_status() == 0
    return kept.view(cache.units, N).cpu().numpy(), scores.view(cache.units, -1).cpu().numpy()


@pytest.mark.parametrize("var", VARIANTS, ids=VAR_IDS)
@pytest.mark.parametrize("factor", [2.0, 0.5])
def test_positive_homogeneity(var, factor):
    """V -> a V with a a power of two (exact in bf16 and in every fp32 step):
    L2 and Norm scores scale by a bit for bit, Dir scores do not change (bit
    for bit too: |v|, |m| and w = v - (|v|/|m|) m all scale exactly); the
    kept set does not change."""
    n, N = 640, 500
    c1 = filled(n, 128, seed=11)
    c2 = vd.Cache(c1.k.clone(), (c1.v.float() * factor).to(torch.bfloat16), c1.len.clone())
    s1, s2 = scores_of(c1, var)[:, :n], scores_of(c2, var)[:, :n]
    if var == vd.VD_SCORE_DIR:
        assert torch.equal(s2, s1)
    else:
        assert torch.equal(s2, s1 * factor)
    k1, _ = evict(c1, N, var)
    k2, _ = evict(c2, N, var)
    assert np.array_equal(k1, k2)


@pytest.mark.parametrize("var", VARIANTS, ids=VAR_IDS)
def test_permutation_equivariance(var):
    """Shuffling the cached rows shuffles the scores with them and keeps the
    same tokens: the kept set is a set of tokens, not of slots."""
    n, N, units = 640, 500, 4
    c1 = filled(n, 128, seed=13, units=units)
    perm = torch.randperm(n, generator=torch.Generator().manual_seed(5))
    c2 = vd.Cache(c1.k[..., perm.cuda(), :].contiguous(), c1.v[..., perm.cuda(), :].contiguous(),
                  c1.len.clone())
    s1 = scores_of(c1, var)[:, :n].double().cpu().numpy()
    s2 = scores_of(c2, var)[:, :n].double().cpu().numpy()
    p = perm.numpy()
    # the mean is summed in another order: it may differ in its last bits
    # (relative 1e-12 of the data), which moves a score by about that much
    assert np.all(np.abs(s2 - s1[:, p]) <= 1e-6 * np.abs(s1[:, p]) + 1e-9)
    k1, _ = evict(c1, N, var)
    k2, _ = evict(c2, N, var)
    for u in range(units):
        diff = np.setxor1d(k1[u], p[k2[u]])           # tokens, in c1's slot numbering
        if diff.size:
            assert np.all(near_tie_band(s1[u], N)[diff]), (u, diff[:8])


def test_translation_invariance_of_l2():
    """v_j -> v_j + c for every j moves the mean by c and leaves every
    deviation v_j - mean unchanged.  With small-integer values and n a power
    of two the mean and every deviation are exact in both runs, so the L2
    scores agree bit for bit (Dir and Norm are not translation invariant)."""
    n, N, units, d = 512, 400, 4, 128
    g = torch.Generator(device="cuda").manual_seed(17)
    cache = new_cache(1, 1, units, n, d)
    v = torch.randint(-8, 9, (units, n, d), generator=g, device="cuda")
    shift = torch.randint(-4, 5, (d,), generator=g, device="cuda")
    units_view(cache.v).copy_(v.to(torch.bfloat16))
    units_view(cache.k).copy_(torch.randint(-8, 9, (units, n, d), generator=g, device="cuda")
                              .to(torch.bfloat16))
    cache.len.fill_(n)
    shifted = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    units_view(shifted.v).copy_((v + shift).to(torch.bfloat16))
    s1 = scores_of(cache, vd.VD_SCORE_L2)[:, :n]
    s2 = scores_of(shifted, vd.VD_SCORE_L2)[:, :n]
    assert torch.equal(s1, s2)
    assert not torch.equal(scores_of(cache, vd.VD_SCORE_NORM)[:, :n],
                           scores_of(shifted, vd.VD_SCORE_NORM)[:, :n])
    k1, _ = evict(cache, N, vd.VD_SCORE_L2)
    k2, _ = evict(shifted, N, vd.VD_SCORE_L2)
    assert np.array_equal(k1, k2)
    # the same tokens' K rows were kept, in the same order
    assert torch.equal(cache.k, shifted.k)


def test_scores_equal_the_uniform_attention_disturbance():
    """Sec. 3.3: under uniform attention the output is the mean of the cached
    values, and removing token j moves it by (mean - v_j) / (n - 1).  Brute
    force in fp64 (recompute the mean without each token) gives
    (n - 1) * |o - o_without_j| = s_j: the GPU's L2 scores match it within the
    parity tolerance and rank the tokens the same way outside near ties."""
    n, d, units, N = 96, 64, 2, 64
    cache = filled(n, d, seed=19, units=units)
    s_gpu = scores_of(cache, vd.VD_SCORE_L2)[:, :n].double().cpu().numpy()
    vals = units_view(cache.v)[:, :n].double().cpu().numpy()
    rows = bits(units_view(cache.v)[:, :n])
    for u in range(units):
        v = vals[u]
        o = v.mean(axis=0)
        disturb = np.array([(n - 1) * np.linalg.norm(o - np.delete(v, j, axis=0).mean(axis=0))
                            for j in range(n)])
        tol = score_tolerance(oracle.L2, disturb, rows[u], o)
        record_error(oracle.L2, s_gpu[u], disturb, tol=tol)
        assert np.all(np.abs(s_gpu[u] - disturb) <= tol)
        top_gpu = np.sort(np.argsort(-s_gpu[u], kind="stable")[:N])
        top_bf = np.sort(np.argsort(-disturb, kind="stable")[:N])
        diff = np.setxor1d(top_gpu, top_bf)
        if diff.size:
            assert np.all(near_tie_band(disturb, N)[diff])
