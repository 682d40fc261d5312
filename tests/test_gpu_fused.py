"""vd_append_evict_block (append and block eviction in one launch) against
vd_append followed by vd_evict_block: identical kept slots, scores,
compacted K/V bytes, running sum and lengths.  The two-call path is the one
the other tests check against the fp64 oracle.  Needs a GB300."""
from __future__ import annotations

import contextlib
import os

import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import new_cache, units_view

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


def setup(d, N, B, lens, seed, cap=None, gen="student_t"):
    cap = cap or N + B
    cache = new_cache(len(lens), 2, 2, cap, d)
    st = wl.TokenStream(gen, cache.units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    us = cache.unit_shape()
    k, v = st.next(B)
    return cache, k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()


def run_both(cache, k_new, v_new, B, N, var, mu):
    us = cache.unit_shape()
    out = []
    for fused in (False, True):
        c = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
        rs = None
        if mu == vd.VD_MU_RUNNING:
            rs = torch.zeros(us + (cache.head_dim,), dtype=torch.float64, device="cuda")
            vd.vd_running_sum_init(c, rs)
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        scores = torch.full(us + (cache.capacity,), float("nan"), device="cuda")
        if fused:
            vd.vd_append_evict_block(c, k_new, v_new, B, N, None, var, mu, rs, kept, scores)
        else:
            vd.vd_append(c, k_new, v_new, B)
            vd.vd_evict_block(c, N, None, B, var, mu, rs, kept, scores)
        assert vd.vd_get_device_status() == 0
        out.append((c, rs, kept, scores))
    return out


def assert_same(a, b):
    (ca, rsa, ka, sa), (cb, rsb, kb, sb) = a, b
    assert torch.equal(ca.len, cb.len)
    assert torch.equal(ka, kb)
    # scores: bit-identical where written (NaN elsewhere in both)
    assert torch.equal(sa.view(torch.int32), sb.view(torch.int32))
    lens = ca.len.cpu().tolist()
    per_seq = ca.n_layer * ca.n_kv_head
    ua, ub = units_view(ca.k), units_view(cb.k)
    va, vb = units_view(ca.v), units_view(cb.v)
    for u in range(ca.units):
        n = lens[u // per_seq]
        assert torch.equal(ua[u, :n].view(torch.int16), ub[u, :n].view(torch.int16)), u
        assert torch.equal(va[u, :n].view(torch.int16), vb[u, :n].view(torch.int16)), u
    if rsa is not None:
        assert torch.equal(rsa, rsb)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("d", [64, 128, 200, 256])
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
def test_fused_equals_append_then_evict(var, d, mu):
    N, B = 160, 48
    # at budget (steady state), partly over (some new rows stay in place),
    # below budget after the append (no eviction)
    lens = [N, N - 20, N - B - 5]
    cache, k_new, v_new = setup(d, N, B, lens, seed=d + 3 * mu + var)
    for c in (None, 2):
        if c is not None and (2 * (d // 8)) % c:
            continue
        with cluster_size(c):
            a, b = run_both(cache, k_new, v_new, B, N, var, mu)
        assert_same(a, b)
        assert a[0].len.cpu().tolist() == [N, N, N - 5]


@pytest.mark.parametrize("cluster", [1, 4, 8])
def test_fused_prefill_shape_and_repeated_events(cluster):
    """Block-processing loop at the benchmark's head dim: five events in a
    row, fused and two-call, stay identical (running mean carried along)."""
    d, N, B = 256, 512, 64
    cache, _, _ = setup(d, N, B, [N, N], seed=41, cap=N + B)
    st = wl.TokenStream("student_t", cache.units, d, device="cuda", seed=42)
    us = cache.unit_shape()
    ca = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    cb = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    rsa = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(ca, rsa)
    rsb = rsa.clone()
    with cluster_size(cluster):
        for _ in range(5):
            k, v = st.next(B)
            k, v = k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()
            ka = torch.empty(us + (N,), dtype=torch.int32, device="cuda")
            kb = torch.empty_like(ka)
            vd.vd_append(ca, k, v, B)
            vd.vd_evict_block(ca, N, None, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rsa, ka)
            vd.vd_append_evict_block(cb, k, v, B, N, None, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rsb, kb)
            assert vd.vd_get_device_status() == 0
            assert torch.equal(ka, kb)
            assert torch.equal(ca.len, cb.len) and int(cb.len[0]) == N
            assert torch.equal(ca.k[..., :N, :].view(torch.int16), cb.k[..., :N, :].view(torch.int16))
            assert torch.equal(ca.v[..., :N, :].view(torch.int16), cb.v[..., :N, :].view(torch.int16))
            assert torch.equal(rsa, rsb)


def test_fused_over_capacity_is_reported_and_untouched():
    d, N, B = 64, 40, 16
    cache, k_new, v_new = setup(d, N, B, [N, N - 10], seed=5, cap=N + 8)   # N + B > capacity
    before_k, before_v = cache.k.clone(), cache.v.clone()
    vd.vd_append_evict_block(cache, k_new, v_new, B, N, None, vd.VD_SCORE_L2, vd.VD_MU_RECOMPUTE)
    assert vd.vd_get_device_status() == 7      # VD_ERR_DEVICE_LEN (first sequence)
    assert int(cache.len[0]) == N               # left untouched
    assert torch.equal(cache.k[0].view(torch.int16), before_k[0].view(torch.int16))
    assert torch.equal(cache.v[0].view(torch.int16), before_v[0].view(torch.int16))
    assert int(cache.len[1]) == N               # the other sequence fitted: N - 10 + 16 -> N


def test_fused_argument_errors():
    cache, k_new, v_new = setup(64, 32, 8, [32], seed=1)
    lib = vd.load_library()
    call = lambda k, v, B: lib.vd_append_evict_block(  # noqa: E731
        cache.ref(), k, v, B, 32, None, 0, 0, None, None, None, None, None, None)
    assert call(k_new.data_ptr(), v_new.data_ptr(), 0) == 1          # B < 1
    assert call(k_new.data_ptr(), None, 8) == 1                      # one buffer missing
    assert call(k_new.data_ptr() + 2, v_new.data_ptr(), 8) == 2      # not 16-byte aligned
    assert int(cache.len[0]) == 32


def run_both_holefill(cache, k_new, v_new, B, N, var, mu, lens):
    us = cache.unit_shape()
    cap = cache.capacity
    out = []
    for fused in (False, True):
        c = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
        pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(c.units).view(
            us + (cap,)).contiguous()
        pos_new = torch.tensor(lens, dtype=torch.int32, device="cuda")  # position of the first new row
        rs = None
        if mu == vd.VD_MU_RUNNING:
            rs = torch.zeros(us + (cache.head_dim,), dtype=torch.float64, device="cuda")
            vd.vd_running_sum_init(c, rs)
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        scores = torch.full(us + (cap,), float("nan"), device="cuda")
        if fused:
            vd.vd_append_evict_block(c, k_new, v_new, B, N, None, var, mu, rs, kept, scores,
                                     pos=pos, pos_first_new=pos_new)
        else:
            vd.vd_append(c, k_new, v_new, B)
            vd.vd_evict_block_holefill(c, N, pos, pos_new, None, B, var, mu, rs, kept, scores)
        assert vd.vd_get_device_status() == 0
        out.append((c, rs, kept, scores, pos))
    return out


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
@pytest.mark.parametrize("d", [128, 200])
def test_fused_holefill_equals_append_then_evict(var, mu, d):
    N, B = 160, 48
    lens = [N, N - 20, N - B - 5]
    cache, k_new, v_new = setup(d, N, B, lens, seed=d + 5 * mu + var)
    for c in (None, 1, 2):
        with cluster_size(c):
            a, b = run_both_holefill(cache, k_new, v_new, B, N, var, mu, lens)
        assert_same(a[:4], b[:4])
        new_lens = a[0].len.cpu().tolist()
        assert new_lens == [N, N, N - 5]
        per_seq = cache.n_layer * cache.n_kv_head
        pa, pb = a[4].view(cache.units, -1), b[4].view(cache.units, -1)
        for u in range(cache.units):
            n = new_lens[u // per_seq]
            assert torch.equal(pa[u, :n], pb[u, :n]), u


def test_fused_holefill_repeated_events():
    """Five hole-fill block events in a row at the benchmark's head dim, fused
    and two-call, stay identical (positions and running mean carried along)."""
    d, N, B = 256, 512, 64
    cache, _, _ = setup(d, N, B, [N, N], seed=51, cap=N + B)
    st = wl.TokenStream("student_t", cache.units, d, device="cuda", seed=52)
    us = cache.unit_shape()
    cap = N + B
    ca = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    cb = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    pa = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(ca.units).view(us + (cap,)).contiguous()
    pb = pa.clone()
    rsa = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(ca, rsa)
    rsb = rsa.clone()
    for e in range(5):
        k, v = st.next(B)
        k, v = k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()
        pn = torch.full((cache.n_seq,), N + e * B, dtype=torch.int32, device="cuda")
        ka = torch.empty(us + (N,), dtype=torch.int32, device="cuda")
        kb = torch.empty_like(ka)
        vd.vd_append(ca, k, v, B)
        vd.vd_evict_block_holefill(ca, N, pa, pn, None, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rsa, ka)
        vd.vd_append_evict_block(cb, k, v, B, N, None, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rsb, kb,
                                 pos=pb, pos_first_new=pn)
        assert vd.vd_get_device_status() == 0
        assert torch.equal(ka, kb) and torch.equal(ca.len, cb.len)
        assert torch.equal(ca.k[..., :N, :].view(torch.int16), cb.k[..., :N, :].view(torch.int16))
        assert torch.equal(ca.v[..., :N, :].view(torch.int16), cb.v[..., :N, :].view(torch.int16))
        assert torch.equal(pa[..., :N], pb[..., :N]) and torch.equal(rsa, rsb)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
@pytest.mark.parametrize("layout", ["ordered", "holefill"])
def test_fused_decode_steps(var, mu, layout):
    """Twelve decode steps, vd_append_evict_decode against vd_append +
    vd_evict_decode(_holefill): identical evicted slots, kept slots, scores,
    cache rows, positions, running sum and lengths; one sequence starts below
    its budget and grows into it."""
    d, N = 128, 96
    lens = [N, N - 3]
    cache, _, _ = setup(d, N, 1, lens, seed=61 + var + 3 * mu, cap=N + 1, gen="drift")
    st = wl.TokenStream("drift", cache.units, d, device="cuda", seed=62)
    us = cache.unit_shape()
    cap = N + 1
    hf = layout == "holefill"
    ca = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    cb = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
    pa = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(ca.units).view(us + (cap,)).contiguous()
    pb = pa.clone()
    rsa = rsb = None
    if mu == vd.VD_MU_RUNNING:
        rsa = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
        vd.vd_running_sum_init(ca, rsa)
        rsb = rsa.clone()
    nextpos = torch.tensor(lens, dtype=torch.int32, device="cuda")
    for step in range(12):
        k, v = st.next(1)
        k, v = k.view(us + (1, d)).contiguous(), v.view(us + (1, d)).contiguous()
        outs = []
        for fused in (False, True):
            c, p, rs = (cb, pb, rsb) if fused else (ca, pa, rsa)
            ev = torch.full(us, -7, dtype=torch.int32, device="cuda")
            kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
            sc = torch.full(us + (cap,), float("nan"), device="cuda")
            hfa = dict(pos=p, pos_first_new=nextpos) if hf else {}
            if fused:
                vd.vd_append_evict_decode(c, k, v, N, None, var, mu, rs, ev, kept, sc, **hfa)
            else:
                vd.vd_append(c, k, v, 1)
                if hf:
                    vd.vd_evict_decode_holefill(c, N, p, nextpos, None, var, mu, rs, ev, kept, sc)
                else:
                    vd.vd_evict_decode(c, N, None, var, mu, rs, ev, kept, sc)
            assert vd.vd_get_device_status() == 0
            outs.append((ev, kept, sc))
        (ea, ka, sa), (eb, kb, sb) = outs
        assert torch.equal(ea, eb) and torch.equal(ka, kb)
        assert torch.equal(sa.view(torch.int32), sb.view(torch.int32))
        assert torch.equal(ca.len, cb.len)
        lens_now = ca.len.cpu().tolist()
        per_seq = ca.n_layer * ca.n_kv_head
        for u in range(ca.units):
            n = lens_now[u // per_seq]
            for x, y in ((ca.k, cb.k), (ca.v, cb.v)):
                assert torch.equal(units_view(x)[u, :n].view(torch.int16),
                                   units_view(y)[u, :n].view(torch.int16)), (step, u)
            if hf:
                assert torch.equal(pa.view(ca.units, -1)[u, :n], pb.view(ca.units, -1)[u, :n])
        if rsa is not None:
            assert torch.equal(rsa, rsb)
        nextpos += 1
    assert ca.len.cpu().tolist() == [N, N]


def test_fused_per_sequence_budgets():
    """Per-sequence budgets (N_dev): block and decode steps, fused against the
    two-call path, including a sequence whose budget lies below its length."""
    d, N, B = 128, 120, 24
    lens = [100, 120, 60, 119]
    Nd = torch.tensor([110, 120, 40, 80], dtype=torch.int32, device="cuda")
    cache, k_new, v_new = setup(d, N, B, lens, seed=71, cap=N + B)
    us = cache.unit_shape()
    res = []
    for fused in (False, True):
        c = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
        rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
        vd.vd_running_sum_init(c, rs)
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        if fused:
            vd.vd_append_evict_block(c, k_new, v_new, B, N, Nd, vd.VD_SCORE_L2, vd.VD_MU_RUNNING,
                                     rs, kept)
        else:
            vd.vd_append(c, k_new, v_new, B)
            vd.vd_evict_block(c, N, Nd, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, kept)
        assert vd.vd_get_device_status() == 0
        # then one decode step with the same budgets
        st = wl.TokenStream("drift", c.units, d, device="cuda", seed=72)
        k1, v1 = st.next(1)
        k1, v1 = k1.view(us + (1, d)).contiguous(), v1.view(us + (1, d)).contiguous()
        ev = torch.full(us, -7, dtype=torch.int32, device="cuda")
        if fused:
            vd.vd_append_evict_decode(c, k1, v1, N, Nd, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, ev)
        else:
            vd.vd_append(c, k1, v1, 1)
            vd.vd_evict_decode(c, N, Nd, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, ev)
        assert vd.vd_get_device_status() == 0
        res.append((c, rs, kept, ev))
    (ca, rsa, ka, ea), (cb, rsb, kb, eb) = res
    assert torch.equal(ca.len, cb.len) and torch.equal(ka, kb) and torch.equal(ea, eb)
    assert torch.equal(rsa, rsb)
    assert ca.len.cpu().tolist() == [110, 120, 40, 80]
    per_seq = ca.n_layer * ca.n_kv_head
    for u in range(ca.units):
        n = ca.len.cpu().tolist()[u // per_seq]
        assert torch.equal(units_view(ca.k)[u, :n].view(torch.int16), units_view(cb.k)[u, :n].view(torch.int16))
        assert torch.equal(units_view(ca.v)[u, :n].view(torch.int16), units_view(cb.v)[u, :n].view(torch.int16))


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("keys", [False, True], ids=["values", "keys"])
@pytest.mark.parametrize("weighted", [False, True], ids=["plain", "weighted"])
@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
def test_fused_scoring_options_match_two_calls(var, keys, weighted, mu):
    """vd_append_evict_block_ex against vd_append + vd_evict_block_ex: the
    key-side rule, attention weights over the new rows' slots, sigma (L2) and
    either mean give bit-identical kept slots, scores, rows, lengths, running
    sums and sigma."""
    d, N, B = 128, 300, 64
    cache, k_new, v_new = setup(d, N, B, [N, N - 40, 100], seed=311 + 7 * var)
    us = cache.unit_shape()
    attn = None
    if weighted:
        g = torch.Generator(device="cuda").manual_seed(3)
        attn = torch.rand(us + (cache.capacity,), generator=g, device="cuda") * 0.9
    out = []
    for fused in (False, True):
        c = vd.Cache(cache.k.clone(), cache.v.clone(), cache.len.clone())
        rs = None
        if mu == vd.VD_MU_RUNNING:
            rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
            vd.vd_running_sum_init_ex(c, keys, rs)
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        scores = torch.full(us + (cache.capacity,), float("nan"), device="cuda")
        sigma = torch.full(us, -1.0, device="cuda") if var == oracle.L2 else None
        if fused:
            vd.vd_append_evict_block_ex(c, k_new, v_new, B, N, None, var, mu, rs, keys, attn,
                                        kept, scores, sigma)
        else:
            vd.vd_append(c, k_new, v_new, B)
            vd.vd_evict_block_ex(c, N, None, B, var, mu, rs, keys, attn, kept, scores, sigma)
        assert vd.vd_get_device_status() == 0
        out.append(((c, rs, kept, scores), sigma))
    assert_same(out[0][0], out[1][0])
    if out[0][1] is not None:
        assert torch.equal(out[0][1], out[1][1])
