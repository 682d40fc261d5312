"""CUDA path (through the C ABI) against the fp64 oracle, step-locked: the
oracle gets the exact pre-eviction bytes of every checked unit at every
checked event.  Needs a GB300 (sm_103a)."""
from __future__ import annotations

import contextlib
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import bits, check_event, check_scores, new_cache, units_view

pytestmark = pytest.mark.gpu

VARS = [oracle.L2, oracle.DIR, oracle.NORM]
VAR_IDS = ["l2", "dir", "norm"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


@contextlib.contextmanager
def cluster_size(c):
    old = os.environ.get("VD_CLUSTER_SIZE")
    if c is None:
        os.environ.pop("VD_CLUSTER_SIZE", None)
    else:
        os.environ["VD_CLUSTER_SIZE"] = str(c)
    try:
        yield
    finally:
        if old is None:
            os.environ.pop("VD_CLUSTER_SIZE", None)
        else:
            os.environ["VD_CLUSTER_SIZE"] = old


def filled_cache(n_seq, L, H, cap, d, lens, gen="gauss_outlier", seed=0, **kw):
    cache = new_cache(n_seq, L, H, cap, d)
    st = wl.TokenStream(gen, cache.units, d, device="cuda", seed=seed, **kw)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    return cache


def evict_and_check(orc, cache, N, B, var, mu, rs=None, units=None, decode=False, N_dev=None):
    """Runs one eviction call and checks the listed units (default: all)."""
    U = cache.units
    per_seq = cache.n_layer * cache.n_kv_head
    idx = list(range(U)) if units is None else list(units)
    it = torch.tensor(idx, device="cuda", dtype=torch.long)
    lens = cache.len.cpu().numpy().copy()
    Ns = N_dev.cpu().numpy() if N_dev is not None else np.full(cache.n_seq, N)
    pre_k = bits(units_view(cache.k)[it])
    pre_v = bits(units_view(cache.v)[it])
    us = cache.unit_shape()
    kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
    scores = torch.full(us + (cache.capacity,), float("nan"), device="cuda")
    evicted = torch.full(us, -7, dtype=torch.int32, device="cuda")
    if decode:
        vd.vd_evict_decode(cache, N, N_dev, var, mu, rs, evicted, kept, scores)
    else:
        vd.vd_evict_block(cache, N, N_dev, B, var, mu, rs, kept, scores)
    assert vd.vd_get_device_status() == 0
    post_k = bits(units_view(cache.k)[it])
    post_v = bits(units_view(cache.v)[it])
    new_lens = cache.len.cpu().numpy()
    kept_h = kept.view(U, N).cpu().numpy()
    sc_h = scores.view(U, cache.capacity).cpu().numpy()
    ev_h = evicted.view(U).cpu().numpy()
    for i, u in enumerate(idx):
        s = u // per_seq
        n, Nb = int(lens[s]), int(Ns[s])
        check_event(orc, var, pre_k[i], pre_v[i], post_k[i], post_v[i], n, Nb,
                    kept_gpu=kept_h[u], scores_gpu=sc_h[u], new_len=int(new_lens[s]))
        if decode:
            if n <= Nb:
                assert ev_h[u] == -1
            else:
                missing = sorted(set(range(n)) - set(kept_h[u][:Nb].tolist()))
                assert [int(ev_h[u])] == missing
    return kept_h


# ---------------------------------------------------------------------------
# scores (vd_score): every variant, head dims incl. non powers of two, ragged n
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("d", [8, 24, 64, 128, 200, 256])
def test_scores_match_oracle(orc, var, d):
    lens = [1, 37, 300, 1000]
    cache = filled_cache(4, 2, 2, 1000, d, lens, seed=d)
    for c in (None, 1, 2, 4):
        with cluster_size(c):
            out = torch.full(cache.unit_shape() + (cache.capacity,), float("nan"), device="cuda")
            vd.vd_score(cache, var, out)
            assert vd.vd_get_device_status() == 0
            o = out.view(cache.units, -1).cpu().numpy()
            v = bits(units_view(cache.v))
            for u in range(cache.units):
                n = lens[u // 4]
                check_scores(orc, var, v[u, :n], o[u, :n])
                assert np.all(np.isnan(o[u, n:])), "rows >= len must stay untouched"


# ---------------------------------------------------------------------------
# one block event, all cluster sizes, both mean modes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
@pytest.mark.parametrize("cluster", [1, 2, 4, 8, 16])
def test_block_event(orc, var, mu, cluster):
    d, N, B = 128, 200, 56
    if 2 * (d // 8) % cluster:
        pytest.skip("cluster does not divide the row")
    lens = [N + B, N + 3, N, 77]          # evict, evict a few, exactly at budget, below budget
    cache = filled_cache(4, 3, 2, N + B, d, lens, seed=cluster)
    rs = None
    if mu == vd.VD_MU_RUNNING:
        # the running sum covers the rows present before this block's B rows
        rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
        cache.len.copy_(torch.tensor([x - B for x in lens], dtype=torch.int32))
        vd.vd_running_sum_init(cache, rs)
        cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    with cluster_size(cluster):
        evict_and_check(orc, cache, N, B, var, mu, rs)
    if rs is not None:
        ref = torch.zeros_like(rs)
        vd.vd_running_sum_init(cache, ref)
        scale = units_view(cache.v).float().abs().sum(dim=1).max().item()
        assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale


# ---------------------------------------------------------------------------
# full tiny prefill (config 0), every event step-locked
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
def test_tiny_prefill_every_event(orc, var, mu):
    _, cfg = wl.config("tiny_prefill")
    d, N, B, T = cfg["head_dim"], cfg["N"], cfg["B"], cfg["T"]
    cache = new_cache(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], N + B, d)
    st = wl.stream_for(cfg)
    rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    events = 0
    for _ in range(T // B):
        k, v = st.next(B)
        vd.vd_append(cache, k.view(cache.unit_shape() + (B, d)), v.view(cache.unit_shape() + (B, d)), B)
        evict_and_check(orc, cache, N, B, var, mu, rs if mu else None)
        events += int(cache.len[0].item() == N)
    assert events >= (T - N) // B


# ---------------------------------------------------------------------------
# decode == block with B = 1, bit for bit
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_decode_equals_block_b1(var):
    d, N = 128, 300
    a = filled_cache(2, 2, 2, N + 1, d, [N + 1, N + 1], seed=5)
    b = vd.Cache(a.k.clone(), a.v.clone(), a.len.clone())
    ka = torch.empty(a.unit_shape() + (N,), dtype=torch.int32, device="cuda")
    kb = torch.empty_like(ka)
    vd.vd_evict_block(a, N, None, 1, var, vd.VD_MU_RECOMPUTE, None, ka, None)
    vd.vd_evict_decode(b, N, None, var, vd.VD_MU_RECOMPUTE, None, None, kb, None)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(ka, kb)
    assert torch.equal(a.k.view(torch.int16), b.k.view(torch.int16))
    assert torch.equal(a.v.view(torch.int16), b.v.view(torch.int16))
    assert torch.equal(a.len, b.len)


# ---------------------------------------------------------------------------
# decode steps with the running mean, checked against recompute
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_decode_steps_running_sum(orc, var):
    d, N = 64, 96
    cache = filled_cache(3, 2, 2, N + 1, d, [N, N, N - 5], seed=11, gen="drift")
    rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(cache, rs)
    st = wl.TokenStream("drift", cache.units, d, seed=12)
    for step in range(40):
        k, v = st.next(1)
        vd.vd_append(cache, k.view(cache.unit_shape() + (1, d)), v.view(cache.unit_shape() + (1, d)), 1)
        evict_and_check(orc, cache, N, 1, var, vd.VD_MU_RUNNING, rs, decode=True)
        if step % 8 == 7:
            ref = torch.zeros_like(rs)
            vd.vd_running_sum_init(cache, ref)
            scale = units_view(cache.v).float().abs().sum(dim=1).max().item()
            assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale
            # and against the oracle's fp64 sum
            vh = bits(units_view(cache.v))
            lens = cache.len.cpu().numpy()
            got = rs.view(cache.units, d).cpu().numpy()
            for u in range(cache.units):
                rows = vh[u, :lens[u // 4]]
                want = orc.sum_rows(rows)
                scale = np.abs(oracle.bits_to_float(rows)).sum(axis=0)
                assert np.all(np.abs(want - got[u]) <= 1e-12 * np.maximum(scale, 1e-30))


# ---------------------------------------------------------------------------
# block then decode events at head dims with the batched score pass (64, 256)
# and without it (96), ragged batch tails, both mean modes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("d", [64, 96, 256])
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
def test_block_then_decode_head_dims(orc, var, d, mu):
    N, B = 150, 37                      # B and the lengths are not multiples of a batch
    lens = [N + B, N + 1, N + 20]
    cache = filled_cache(3, 2, 2, N + B, d, lens, seed=d + 7 * mu, gen="student_t")
    rs = None
    if mu == vd.VD_MU_RUNNING:
        rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
        cache.len.copy_(torch.tensor([x - B for x in lens], dtype=torch.int32))
        vd.vd_running_sum_init(cache, rs)
        cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    for c in (None, 2):
        if c is not None and 2 * (d // 8) % c:
            continue
        work = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
        wrs = rs.clone() if rs is not None else None
        with cluster_size(c):
            evict_and_check(orc, work, N, B, var, mu, wrs)
            # one decode step on the compacted cache
            st = wl.TokenStream("student_t", work.units, d, device="cuda", seed=d + 1)
            k, v = st.next(1)
            us = work.unit_shape()
            vd.vd_append(work, k.view(us + (1, d)).contiguous(), v.view(us + (1, d)).contiguous(), 1)
            evict_and_check(orc, work, N, 1, var, mu, wrs, decode=True)
        if wrs is not None:
            ref = torch.zeros_like(wrs)
            vd.vd_running_sum_init(work, ref)
            scale = units_view(work.v).float().abs().sum(dim=1).max().item()
            assert torch.max(torch.abs(ref - wrs)).item() <= 1e-12 * scale


# ---------------------------------------------------------------------------
# ties, duplicates, degenerate caches, N extremes, poisoned tails
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_ties_duplicates_and_small_integers(orc, var):
    d, N, B = 64, 120, 40
    for kw in (dict(dup_fraction=0.3), dict(small_int=True), dict(small_int=True, dup_fraction=0.5)):
        cache = filled_cache(2, 2, 2, N + B, d, [N + B, N + B], seed=3, **kw)
        evict_and_check(orc, cache, N, B, var, vd.VD_MU_RECOMPUTE)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_all_rows_equal_keeps_first_n(var):
    d, n, N = 32, 50, 20
    cache = new_cache(1, 1, 2, n, d)
    row = torch.randn(d, device="cuda").to(torch.bfloat16)
    cache.k.copy_(torch.randn_like(cache.k, dtype=torch.float32).to(torch.bfloat16))
    cache.v[:] = row
    cache.len.fill_(n)
    kept = torch.empty(1, 1, 2, N, dtype=torch.int32, device="cuda")
    vd.vd_evict_block(cache, N, None, 0, var, vd.VD_MU_RECOMPUTE, None, kept, None)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(kept.cpu(), torch.arange(N, dtype=torch.int32).expand(1, 1, 2, N))
    assert int(cache.len[0]) == N


@pytest.mark.parametrize("N", [1, 2, 499])
def test_budget_extremes(orc, N):
    n, d = 500, 128
    cache = filled_cache(1, 2, 2, n, d, [n], seed=N)
    evict_and_check(orc, cache, N, 0, oracle.L2, vd.VD_MU_RECOMPUTE)


def test_poisoned_tail_never_read(orc):
    d, N, B, cap = 128, 100, 30, 200
    cache = filled_cache(2, 2, 2, cap, d, [N + B, N + B], seed=21)
    clean = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    nan = torch.tensor(0x7FC0, dtype=torch.int16).view(torch.bfloat16)
    cache.v[..., N + B:, :] = nan
    cache.k[..., N + B:, :] = nan
    for c in (cache, clean):
        vd.vd_evict_block(c, N, None, B, oracle.L2, vd.VD_MU_RECOMPUTE, None, None, None)
    assert vd.vd_get_device_status() == 0
    assert torch.equal(cache.v[..., :N, :].view(torch.int16), clean.v[..., :N, :].view(torch.int16))
    assert torch.equal(cache.k[..., :N, :].view(torch.int16), clean.k[..., :N, :].view(torch.int16))
    # the poisoned slots past the old length are left alone
    assert torch.equal(cache.v[..., N + B:, :].view(torch.int16),
                       torch.full_like(cache.v[..., N + B:, :].view(torch.int16), 0x7FC0))


def test_ragged_lengths_and_per_sequence_budgets(orc):
    d, cap = 128, 700
    lens = [700, 650, 100, 699, 3]
    Ns = torch.tensor([600, 650, 50, 1, 3], dtype=torch.int32, device="cuda")
    cache = filled_cache(5, 2, 3, cap, d, lens, seed=8)
    evict_and_check(orc, cache, 650, 0, oracle.L2, vd.VD_MU_RECOMPUTE, N_dev=Ns)


def test_block_equals_one_shot_standard_eviction(orc):
    """B = T recovers standard eviction (Sec. 2.2): one event over the whole
    prompt equals the oracle's one-shot top-N."""
    d, T, N = 64, 1536, 256
    cache = filled_cache(1, 2, 2, T, d, [T], seed=13)
    evict_and_check(orc, cache, N, T, oracle.L2, vd.VD_MU_RECOMPUTE)


# ---------------------------------------------------------------------------
# device-side anomalies are reported, never trapped, and leave units untouched
# ---------------------------------------------------------------------------
def test_nonfinite_score_is_reported():
    d, n, N = 64, 80, 60
    cache = filled_cache(1, 1, 1, n, d, [n], seed=2)
    cache.v[0, 0, 0, 5, 3] = float("nan")
    vd.vd_evict_block(cache, N, None, 0, oracle.L2, vd.VD_MU_RECOMPUTE, None, None, None)
    assert vd.vd_get_device_status() == 4   # VD_ERR_NONFINITE
    assert vd.vd_get_device_status() == 0   # cleared by the read


def test_decode_over_budget_is_reported_and_untouched():
    d, N = 64, 40
    cache = filled_cache(1, 1, 2, N + 5, d, [N + 3], seed=4)
    before = cache.v.clone()
    vd.vd_evict_decode(cache, N, None, oracle.L2, vd.VD_MU_RECOMPUTE, None, None, None, None)
    assert vd.vd_get_device_status() == 8   # VD_ERR_DEVICE_BUDGET
    assert torch.equal(before.view(torch.int16), cache.v.view(torch.int16))
    assert int(cache.len[0]) == N + 3


def test_len_beyond_capacity_is_reported():
    d = 64
    cache = filled_cache(1, 1, 1, 64, d, [64], seed=6)
    cache.len.fill_(65)
    out = torch.zeros(1, 1, 1, 64, device="cuda")
    vd.vd_score(cache, oracle.L2, out)
    assert vd.vd_get_device_status() == 7   # VD_ERR_DEVICE_LEN
    assert torch.all(out == 0)


def test_append_and_overflow():
    d, cap, B = 64, 100, 30
    cache = filled_cache(2, 1, 2, cap, d, [10, 80], seed=9)
    before = cache.v.clone()
    k = torch.randn(2, 1, 2, B, d, device="cuda").to(torch.bfloat16)
    v = torch.randn(2, 1, 2, B, d, device="cuda").to(torch.bfloat16)
    vd.vd_append(cache, k, v, B)
    assert vd.vd_get_device_status() == 7   # sequence 1 would overflow
    assert cache.len.tolist() == [10 + B, 80]
    assert torch.equal(cache.v[0, :, :, 10:10 + B].view(torch.int16), v[0].view(torch.int16))
    assert torch.equal(cache.k[0, :, :, 10:10 + B].view(torch.int16), k[0].view(torch.int16))
    assert torch.equal(cache.v[1].view(torch.int16), before[1].view(torch.int16))


def test_running_sum_init_matches_oracle(orc):
    d = 256
    cache = filled_cache(2, 2, 2, 3000, d, [3000, 17], seed=10, gen="student_t")
    rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(cache, rs)
    v = bits(units_view(cache.v))
    got = rs.view(cache.units, d).cpu().numpy()
    for u in range(cache.units):
        n = [3000, 17][u // 4]
        want = orc.sum_rows(v[u, :n])
        scale = np.abs(oracle.bits_to_float(v[u, :n])).sum(axis=0)
        assert np.all(np.abs(got[u] - want) <= 1e-12 * np.maximum(scale, 1e-30))
