"""The scoring options of vd_score_ex / vd_evict_block_ex against the fp64
oracle: key-side rules (the same scores on K), attention-weighted scores
(App. A Eq. app_fastcaote) and the per-unit dispersion sigma (Sec. 3.1).
Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import (RTOL, bits, near_tie_band, new_cache, record_error, score_tolerance,
                    units_view, weighted_tolerance)

pytestmark = pytest.mark.gpu
VARS = [oracle.L2, oracle.DIR, oracle.NORM]
VAR_IDS = ["l2", "dir", "norm"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def filled(n_seq, L, H, cap, d, lens, seed, gen="gauss_outlier"):
    cache = new_cache(n_seq, L, H, cap, d)
    st = wl.TokenStream(gen, cache.units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    return cache


def check_scored_event(s_ora, tol, pre_k, pre_v, post_k, post_v, n, N, kept_gpu, scores_gpu,
                       var=None, tag=""):
    """One unit: GPU scores within tol of the oracle's, the same kept set
    outside near ties, bit-exact gathers of K and V."""
    if n <= N:
        assert np.array_equal(post_v[:n], pre_v[:n]) and np.array_equal(post_k[:n], pre_k[:n])
        return
    err = np.abs(scores_gpu[:n].astype(np.float64) - s_ora)
    record_error(var, scores_gpu[:n], s_ora, tag, tol)
    assert np.all(err <= tol), f"worst score error {err.max():.3e}"
    kept_ora = orc_select(s_ora, N)
    kg = np.asarray(kept_gpu[:N], np.int64)
    assert np.all(np.diff(kg) > 0)
    diff = np.setxor1d(kg, kept_ora)
    if diff.size:
        assert np.all(near_tie_band(s_ora, N)[diff]), f"kept sets differ at {diff[:8]}"
    assert np.array_equal(post_k[:N], pre_k[:n][kg]) and np.array_equal(post_v[:N], pre_v[:n][kg])


_ORC = None


def orc_select(s, N):
    return _ORC.select_top_n(s, N)


def run_ex(orc, cache, N, B, var, score_keys, attn):
    global _ORC
    _ORC = orc
    U, cap = cache.units, cache.capacity
    per_seq = cache.n_layer * cache.n_kv_head
    lens = cache.len.cpu().numpy().copy()
    pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    us = cache.unit_shape()
    kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
    scores = torch.full(us + (cap,), float("nan"), device="cuda")
    vd.vd_evict_block_ex(cache, N, None, B, var, vd.VD_MU_RECOMPUTE, None, score_keys, attn, kept,
                         scores)
    assert vd.vd_get_device_status() == 0
    post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    kh, sh = kept.view(U, N).cpu().numpy(), scores.view(U, cap).cpu().numpy()
    a_h = attn.view(U, cap).cpu().numpy().astype(np.float64) if attn is not None else None
    for u in range(U):
        n = int(lens[u // per_seq])
        src = pre_k[u, :n] if score_keys else pre_v[u, :n]
        if a_h is None:
            s_ora = orc.scores(src, var)
            tol = score_tolerance(var, s_ora, src, orc.mean(src))
        else:
            s_ora = orc.scores_weighted(src, a_h[u, :n], var)
            base = orc.scores(src, var)
            f = a_h[u, :n] / (1.0 - a_h[u, :n])
            tol = weighted_tolerance(var, s_ora, base, src, orc.mean(src), f)
        check_scored_event(s_ora, tol, pre_k[u], pre_v[u], post_k[u], post_v[u], n, N, kh[u], sh[u],
                           var, ("_k" if score_keys else "") + ("_w" if a_h is not None else ""))


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 4])
def test_key_side_eviction(orc, var, cluster, monkeypatch):
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 128, 300, 64
    cache = filled(3, 2, 2, N + B, d, [N + B, N + 10, 50], seed=17 + cluster)
    run_ex(orc, cache, N, B, var, True, None)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 2])
def test_attention_weighted_eviction(orc, var, cluster, monkeypatch):
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 64, 200, 40
    cache = filled(2, 2, 2, N + B, d, [N + B, N + 7], seed=23 + cluster)
    g = torch.Generator(device="cuda").manual_seed(5)
    attn = torch.rand(cache.unit_shape() + (N + B,), generator=g, device="cuda") * 0.9
    attn[..., ::17] = 0.0                     # tokens with no attention score 0
    run_ex(orc, cache, N, B, var, False, attn)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 2])
def test_negative_zero_weight_and_nan_rank(orc, var, cluster, monkeypatch):
    """A weight of -0 gives the score -0, which ranks with the zero scores
    (ties to the lower slot), and a NaN score (a weight of 1, reported as
    VD_ERR_NONFINITE) ranks below every zero score, so it is evicted first:
    the kept set equals the oracle's, which orders NaN last."""
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, n, N = 64, 120, 95
    cache = filled(1, 1, 2, n, d, [n], seed=31 + cluster)
    attn = torch.full(cache.unit_shape() + (n,), 0.3, device="cuda")
    attn[..., :40] = 0.0
    attn[..., 0:40:2] = -0.0                  # 20 tokens weighted -0
    attn[..., 1:40:4] = 1.0                   # 10 tokens with a NaN score
    pre_v = bits(units_view(cache.v))
    kept = torch.full(cache.unit_shape() + (N,), -7, dtype=torch.int32, device="cuda")
    scores = torch.full(cache.unit_shape() + (n,), float("nan"), device="cuda")
    vd.vd_evict_block_ex(cache, N, variant=var, attn=attn, kept_idx_out=kept, scores_out=scores)
    assert vd.vd_get_device_status() == 4     # VD_ERR_NONFINITE: the NaN scores
    a_h = attn.view(2, n).cpu().numpy().astype(np.float64)
    assert np.signbit(a_h[0, 0]) and a_h[0, 0] == 0.0
    kh = kept.view(2, N).cpu().numpy()
    sh = scores.view(2, n).cpu().numpy()
    for u in range(2):
        s_ora = orc.scores_weighted(pre_v[u, :n], a_h[u], var)
        want = orc.select_top_n(s_ora, N)
        assert np.array_equal(kh[u], want), (u, np.setxor1d(kh[u], want))
        assert not np.any(np.isin(np.arange(1, 40, 4), kh[u]))   # every NaN evicted
        # the zero-weighted tokens report a zero score, the NaN ones NaN
        assert np.all(sh[u, :40][np.isnan(s_ora[:40])] != sh[u, :40][np.isnan(s_ora[:40])])
        assert np.all(sh[u, 0:40:2] == 0.0)


def test_uniform_attention_keeps_the_valuediff_set(orc):
    """App. A: with a_j = 1/n the weighted rule ranks like ValueDiff."""
    d, N, n = 128, 150, 200
    cache = filled(1, 2, 2, n, d, [n], seed=3)
    ref = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    attn = torch.full(cache.unit_shape() + (n,), 1.0 / n, device="cuda")
    ka = torch.empty(cache.unit_shape() + (N,), dtype=torch.int32, device="cuda")
    kb = torch.empty_like(ka)
    vd.vd_evict_block_ex(cache, N, attn=attn, kept_idx_out=ka)
    vd.vd_evict_block(ref, N, kept_idx_out=kb)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(ka, kb)


@pytest.mark.parametrize("keys", [False, True], ids=["sigma_v", "sigma_k"])
@pytest.mark.parametrize("cluster", [1, 2, 4])
def test_dispersion_matches_oracle(orc, keys, cluster, monkeypatch):
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d = 128
    lens = [2048, 777, 1]
    cache = filled(3, 2, 2, 2048, d, lens, seed=41, gen="student_t")
    out = torch.full(cache.unit_shape(), -1.0, device="cuda")
    vd.vd_score_ex(cache, vd.VD_SCORE_L2, keys, None, out)
    assert vd.vd_get_device_status() == 0
    src = bits(units_view(cache.k if keys else cache.v))
    got = out.view(-1).cpu().numpy()
    for u in range(cache.units):
        n = lens[u // 4]
        want = orc.dispersion(src[u, :n])
        assert abs(got[u] - want) <= 1e-5 * want + 1e-6, (u, got[u], want)


@pytest.mark.parametrize("keys", [False, True], ids=["v", "k"])
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 2, 4])
def test_score_ex_running_mean(orc, keys, var, cluster, monkeypatch):
    """vd_score_ex with the mean taken from a running sum (the rows read
    once): scores (and sigma, for L2) match the oracle on the current rows,
    both right after the sum is seeded and after an eviction carried it; the
    sum is only read; rows at or above len are not written."""
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 128, 300, 64
    cache = filled(3, 2, 2, N + B, d, [N, N - 40, 1], seed=71 + cluster, gen="student_t")
    us = cache.unit_shape()
    per_seq = cache.n_layer * cache.n_kv_head
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init_ex(cache, keys, rs)
    st = wl.TokenStream("gauss_outlier", cache.units, d, device="cuda", seed=72)
    for stage in range(2):
        if stage == 1:  # one block event with the running mean carries the sum
            k, v = st.next(B)
            vd.vd_append(cache, k.view(us + (B, d)), v.view(us + (B, d)), B)
            vd.vd_evict_block_ex(cache, N, None, B, var, vd.VD_MU_RUNNING, rs, keys)
        lens = cache.len.cpu().numpy().copy()
        rs_before = rs.clone()
        sc = torch.full(us + (N + B,), float("nan"), device="cuda")
        sig = torch.full(us, -1.0, device="cuda") if var == oracle.L2 else None
        vd.vd_score_ex(cache, var, keys, sc, sig, mu=vd.VD_MU_RUNNING, running_sum=rs)
        assert vd.vd_get_device_status() == 0
        assert torch.equal(rs, rs_before)
        src = bits(units_view(cache.k if keys else cache.v))
        sh = sc.view(cache.units, -1).cpu().numpy()
        for u in range(cache.units):
            n = int(lens[u // per_seq])
            s_ora = orc.scores(src[u, :n], var)
            tol = score_tolerance(var, s_ora, src[u, :n], orc.mean(src[u, :n]))
            err = np.abs(sh[u, :n].astype(np.float64) - s_ora)
            record_error(var, sh[u, :n], s_ora, "_k" if keys else "", tol)
            assert np.all(err <= tol), (stage, u, float(err.max()))
            assert np.all(np.isnan(sh[u, n:]))
            if sig is not None:
                want = orc.dispersion(src[u, :n])
                got = float(sig.view(-1)[u].item())
                assert abs(got - want) <= 1e-5 * want + 1e-6, (stage, u, got, want)


@pytest.mark.parametrize("keys", [False, True], ids=["sigma_v", "sigma_k"])
@pytest.mark.parametrize("cluster", [1, 2, 4])
@pytest.mark.parametrize("weighted", [False, True], ids=["plain", "weighted"])
def test_dispersion_by_product_of_eviction(orc, keys, cluster, weighted, monkeypatch):
    """sigma from the eviction's own score pass: the pre-eviction rows of
    every unit that evicted, untouched elsewhere; the eviction itself is
    unchanged by asking for it."""
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 128, 300, 64
    lens = [N + B, N + 5, 100]
    cache = filled(3, 2, 2, N + B, d, lens, seed=61 + cluster, gen="student_t")
    ref = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    pre = bits(units_view(cache.k if keys else cache.v))
    attn = None
    if weighted:
        g = torch.Generator(device="cuda").manual_seed(9)
        attn = torch.rand(cache.unit_shape() + (N + B,), generator=g, device="cuda") * 0.9
    out = torch.full(cache.unit_shape(), -1.0, device="cuda")
    ka = torch.empty(cache.unit_shape() + (N,), dtype=torch.int32, device="cuda")
    kb = torch.empty_like(ka)
    vd.vd_evict_block_ex(cache, N, score_keys=keys, attn=attn, kept_idx_out=ka,
                         dispersion_out=out)
    vd.vd_evict_block_ex(ref, N, score_keys=keys, attn=attn, kept_idx_out=kb)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(ka, kb)
    assert torch.equal(cache.k, ref.k) and torch.equal(cache.v, ref.v)
    got = out.view(-1).cpu().numpy()
    for u in range(cache.units):
        n = lens[u // 4]
        if n <= N:
            assert got[u] == -1.0
            continue
        want = orc.dispersion(pre[u, :n])
        assert abs(got[u] - want) <= 1e-5 * want + 1e-6, (u, got[u], want)


@pytest.mark.parametrize("cluster", [1, 4])
def test_dispersion_by_product_running_mean(orc, cluster, monkeypatch):
    """With the running-sum mean (S / n) the by-product is the same sigma."""
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 256, 400, 48
    cache = filled(2, 1, 2, N + B, d, [N, N], seed=71 + cluster)
    rs = torch.empty(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(cache, rs)
    cache.len.fill_(N + B)                  # the next B rows were already written
    pre = bits(units_view(cache.v))
    out = torch.full(cache.unit_shape(), -1.0, device="cuda")
    vd.vd_evict_block_ex(cache, N, None, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs,
                         dispersion_out=out)
    assert vd.vd_get_device_status() == 0
    got = out.view(-1).cpu().numpy()
    for u in range(cache.units):
        want = orc.dispersion(pre[u, :N + B])
        assert abs(got[u] - want) <= 1e-5 * want + 1e-6, (u, got[u], want)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 4])
def test_key_side_running_mean(orc, var, cluster, monkeypatch):
    """The key-side rule with the running mean: a running sum of K rows (seeded
    by vd_running_sum_init_ex) carried over block events; each event matches
    the oracle on K, and the sum stays the K rows' sum."""
    global _ORC
    _ORC = orc
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 128, 300, 64
    cache = filled(2, 2, 2, N + B, d, [N, N - 30], seed=91 + cluster)
    us = cache.unit_shape()
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init_ex(cache, True, rs)
    st = wl.TokenStream("gauss_outlier", cache.units, d, device="cuda", seed=92)
    per_seq = cache.n_layer * cache.n_kv_head
    for event in range(3):
        k, v = st.next(B)
        vd.vd_append(cache, k.view(us + (B, d)), v.view(us + (B, d)), B)
        lens = cache.len.cpu().numpy().copy()
        pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        scores = torch.full(us + (N + B,), float("nan"), device="cuda")
        vd.vd_evict_block_ex(cache, N, None, B, var, vd.VD_MU_RUNNING, rs, True, None, kept,
                             scores)
        assert vd.vd_get_device_status() == 0
        post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
        kh, sh = kept.view(cache.units, N).cpu().numpy(), scores.view(cache.units, -1).cpu().numpy()
        for u in range(cache.units):
            n = int(lens[u // per_seq])
            s_ora = orc.scores(pre_k[u, :n], var)
            tol = score_tolerance(var, s_ora, pre_k[u, :n], orc.mean(pre_k[u, :n]))
            check_scored_event(s_ora, tol, pre_k[u], pre_v[u], post_k[u], post_v[u], n, N,
                               kh[u], sh[u], var, "_k")
        ref = torch.zeros_like(rs)
        vd.vd_running_sum_init_ex(cache, True, ref)
        scale = units_view(cache.k).float().abs().sum(dim=1).max().item()
        assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale


def test_option_errors():
    cache = filled(1, 1, 1, 64, 64, [64], seed=1)
    with pytest.raises(vd.VdError) as e:
        vd.vd_score_ex(cache, vd.VD_SCORE_DIR, False, None,
                       torch.zeros(1, 1, 1, device="cuda"))
    assert e.value.code == 1                  # sigma is defined on L2 distances
    with pytest.raises(vd.VdError) as e:
        vd.vd_score_ex(cache, vd.VD_SCORE_L2, False, torch.zeros(1, 1, 1, 64, device="cuda"),
                       mu=vd.VD_MU_RUNNING)
    assert e.value.code == 1                  # a running mean needs its sum
    with pytest.raises(vd.VdError) as e:
        vd.vd_evict_block_ex(cache, 32, variant=vd.VD_SCORE_NORM,
                             dispersion_out=torch.zeros(1, 1, 1, device="cuda"))
    assert e.value.code == 1
    attn = torch.full((1, 1, 1, 64), 0.5, device="cuda")
    attn[..., 3] = 1.0                        # a weight of 1: infinite factor
    vd.vd_evict_block_ex(cache, 32, attn=attn)
    assert vd.vd_get_device_status() == 4


@pytest.mark.parametrize("var", [oracle.L2, oracle.NORM], ids=["l2", "norm"])
@pytest.mark.parametrize("d", [64, 128, 256])
@pytest.mark.parametrize("cluster", [1, 2, 4])
def test_score_only_bulk_ring_matches_the_eviction_score_pass(var, d, cluster, monkeypatch):
    """vd_score at head dims 64/128/256 streams its rows through bulk copies;
    the eviction kernel streams them through per-thread asynchronous copies.
    With the same cluster size (so each CTA sums and scores the same rows)
    the mean and every score are bit-identical."""
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    n = 1500                                   # several 32 KB stages and a ragged last one
    cache = filled(2, 2, 2, n, d, [n, n - 333], seed=91 + d)
    sc = torch.full(cache.unit_shape() + (n,), float("nan"), device="cuda")
    vd.vd_score(cache, var, sc)
    ev = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    sc2 = torch.full_like(sc, float("nan"))
    vd.vd_evict_block(ev, n - 400, None, 0, var, vd.VD_MU_RECOMPUTE, None, None, sc2)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(sc.nan_to_num(-1.0), sc2.nan_to_num(-1.0))
