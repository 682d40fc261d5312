"""The short-cache kernel (one CTA per unit, the unit's rows in shared memory,
one launch per event including the length update) against the fp64 oracle,
step-locked, and against the fused kernel on the same inputs
(VD_SMALL_PATH=0 forces the latter).  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from test_gpu_parity import evict_and_check, filled_cache
from vd_gpu import bits, near_tie_band, units_view

pytestmark = pytest.mark.gpu

VARS = [oracle.L2, oracle.DIR, oracle.NORM]
VAR_IDS = ["l2", "dir", "norm"]
MUS = [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING]
MU_IDS = ["recompute", "running"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def running_sum_of(cache, rows_per_seq):
    """fp64 running sums of the first rows_per_seq[s] rows of every unit."""
    rs = torch.zeros(cache.unit_shape() + (cache.head_dim,), dtype=torch.float64, device="cuda")
    saved = cache.len.clone()
    cache.len.copy_(torch.tensor(rows_per_seq, dtype=torch.int32))
    vd.vd_running_sum_init(cache, rs)
    cache.len.copy_(saved)
    return rs


def check_running_sum(cache, rs):
    ref = torch.zeros_like(rs)
    vd.vd_running_sum_init(cache, ref)
    scale = units_view(cache.v).float().abs().sum(dim=1).max().item()
    assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale


# ---------------------------------------------------------------------------
# block events: every rule and mean mode, ragged lengths, per-sequence
# budgets, cluster sizes 1..16 (units per sequence), head dims 8..128
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", MUS, ids=MU_IDS)
@pytest.mark.parametrize("shape", [(1, 1, 64, 160), (2, 3, 128, 120), (1, 16, 8, 700),
                                   (3, 2, 24, 300)], ids=["1x1", "2x3", "1x16", "3x2"])
def test_block_event_matches_oracle(orc, var, mu, shape):
    L, H, d, cap = shape
    N, B = cap * 2 // 3, cap // 3
    lens = [cap, N + 1, N, B + 2][: 4 if L * H <= 4 else 3]   # running mode needs n >= B
    n_seq = len(lens)
    cache = filled_cache(n_seq, L, H, cap, d, lens, seed=L * 7 + H + d)
    rs = running_sum_of(cache, [max(0, x - B) for x in lens]) if mu else None
    Ns = torch.tensor([N, N - 3, N, 2][:n_seq], dtype=torch.int32, device="cuda")
    evict_and_check(orc, cache, N, B, var, mu, rs, N_dev=Ns)
    if rs is not None:
        check_running_sum(cache, rs)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", MUS, ids=MU_IDS)
def test_decode_steps(orc, var, mu):
    d, N = 64, 200
    cache = filled_cache(2, 2, 3, N + 1, d, [N, N - 4], seed=41, gen="drift")
    rs = running_sum_of(cache, [N, N - 4]) if mu else None
    st = wl.TokenStream("drift", cache.units, d, seed=42)
    us = cache.unit_shape()
    for step in range(12):
        k, v = st.next(1)
        vd.vd_append(cache, k.view(us + (1, d)).contiguous(), v.view(us + (1, d)).contiguous(), 1)
        evict_and_check(orc, cache, N, 1, var, mu, rs, decode=True)
    if rs is not None:
        check_running_sum(cache, rs)


# ---------------------------------------------------------------------------
# the fused append: the kernel reads the new rows from the staging buffers
# and sets the lengths itself (including sequences that do not evict)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("mu", MUS, ids=MU_IDS)
@pytest.mark.parametrize("decode", [False, True], ids=["block", "decode"])
def test_fused_append_matches_two_calls(var, mu, decode):
    d, N = 64, 128
    B = 1 if decode else 32
    cap = N + B
    lens = [N, N - B, N - 1] if not decode else [N, N - 1, N - 3]
    a = filled_cache(3, 1, 2, cap, d, lens, seed=51 + B)
    b = vd.Cache(a.k.clone(), a.v.clone(), a.len.clone())
    ra = running_sum_of(a, lens) if mu else None
    rb = ra.clone() if ra is not None else None
    st = wl.TokenStream("gauss_outlier", a.units, d, seed=52)
    k, v = st.next(B)
    us = a.unit_shape()
    k, v = k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()
    outs = []
    for c, r, fused in ((a, ra, True), (b, rb, False)):
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        sc = torch.full(us + (cap,), float("nan"), device="cuda")
        ev = torch.full(us, -7, dtype=torch.int32, device="cuda")
        if fused and decode:
            vd.vd_append_evict_decode(c, k, v, N, None, var, mu, r, ev, kept, sc)
        elif fused:
            vd.vd_append_evict_block(c, k, v, B, N, None, var, mu, r, kept_idx_out=kept,
                                     scores_out=sc)
        else:
            vd.vd_append(c, k, v, B)
            if decode:
                vd.vd_evict_decode(c, N, None, var, mu, r, ev, kept, sc)
            else:
                vd.vd_evict_block(c, N, None, B, var, mu, r, kept, sc)
        assert vd.vd_get_device_status() == 0
        outs.append((kept, sc, ev))
    assert torch.equal(a.len, b.len)
    assert a.len.tolist() == [min(x + B, N) for x in lens]
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1].nan_to_num(-1.0), outs[1][1].nan_to_num(-1.0))
    if decode:
        assert torch.equal(outs[0][2], outs[1][2])
    for s, n in enumerate(a.len.tolist()):
        assert torch.equal(a.k[s, ..., :n, :].view(torch.int16), b.k[s, ..., :n, :].view(torch.int16))
        assert torch.equal(a.v[s, ..., :n, :].view(torch.int16), b.v[s, ..., :n, :].view(torch.int16))
    if ra is not None:
        assert torch.equal(ra, rb)
        check_running_sum(a, ra)


# ---------------------------------------------------------------------------
# the same event through the fused kernel: same kept sets outside near ties,
# same compacted rows where the sets agree, scores within the tolerance
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_agrees_with_the_fused_kernel(orc, var, monkeypatch):
    d, N, B = 64, 100, 40
    lens = [N + B, N + 9]
    base = filled_cache(2, 2, 2, N + B, d, lens, seed=61, dup_fraction=0.1)
    results = []
    for small in ("1", "0"):
        monkeypatch.setenv("VD_SMALL_PATH", small)
        c = vd.Cache(base.k.clone(), base.v.clone(), base.len.clone())
        kept = torch.full(c.unit_shape() + (N,), -7, dtype=torch.int32, device="cuda")
        sc = torch.full(c.unit_shape() + (N + B,), float("nan"), device="cuda")
        vd.vd_evict_block(c, N, None, B, var, vd.VD_MU_RECOMPUTE, None, kept, sc)
        assert vd.vd_get_device_status() == 0
        results.append((c, kept.view(c.units, N).cpu().numpy(), sc.view(c.units, -1).cpu().numpy()))
    (c1, k1, s1), (c2, k2, s2) = results
    assert torch.equal(c1.len, c2.len)
    pre_v = bits(units_view(base.v))
    for u in range(base.units):
        n = lens[u // 4]
        s_ora = orc.scores(pre_v[u, :n], var)
        band = near_tie_band(s_ora, N)
        diff = np.setxor1d(k1[u], k2[u])
        assert np.all(band[diff]), (u, diff)
        assert np.all(np.abs(s1[u, :n].astype(np.float64) - s2[u, :n]) <= 2e-5 * s_ora + 2e-11)
        if diff.size == 0:
            assert torch.equal(units_view(c1.v)[u, :N].view(torch.int16),
                               units_view(c2.v)[u, :N].view(torch.int16))
            assert torch.equal(units_view(c1.k)[u, :N].view(torch.int16),
                               units_view(c2.k)[u, :N].view(torch.int16))


def test_tiny_prefill_every_event_both_kernels(orc, monkeypatch):
    """The smallest workload, every event, with and without the short-cache
    kernel: identical kept lists and caches (no near ties in this stream)."""
    _, cfg = wl.config("tiny_prefill")
    d, N, B, T = cfg["head_dim"], cfg["N"], cfg["B"], cfg["T"]
    caches = []
    for small in ("1", "0"):
        monkeypatch.setenv("VD_SMALL_PATH", small)
        cache = vd.Cache.empty(1, 1, 2, N + B, d)
        st = wl.stream_for(cfg)
        rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
        kept_all = []
        for _ in range(T // B):
            k, v = st.next(B)
            us = cache.unit_shape()
            kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
            vd.vd_append_evict_block(cache, k.view(us + (B, d)).contiguous(),
                                     v.view(us + (B, d)).contiguous(), B, N, None,
                                     vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, kept_idx_out=kept)
            kept_all.append(kept.clone())
        assert vd.vd_get_device_status() == 0
        caches.append((cache, kept_all, rs))
    (a, ka, ra), (b, kb, rb) = caches
    assert all(torch.equal(x, y) for x, y in zip(ka, kb))
    assert torch.equal(a.k.view(torch.int16), b.k.view(torch.int16))
    assert torch.equal(a.v.view(torch.int16), b.v.view(torch.int16))
    assert torch.equal(a.len, b.len) and int(a.len[0]) == N
    assert torch.max(torch.abs(ra - rb)).item() <= 1e-12 * ra.abs().max().item()


# ---------------------------------------------------------------------------
# anomalies: the same status codes as the fused kernel, lengths untouched
# ---------------------------------------------------------------------------
def test_decode_over_budget_and_bad_length():
    d, N = 64, 40
    cache = filled_cache(2, 1, 2, N + 5, d, [N + 3, N + 1], seed=71)
    before_v = cache.v.clone()
    vd.vd_evict_decode(cache, N, None, oracle.L2, vd.VD_MU_RECOMPUTE, None, None, None, None)
    assert vd.vd_get_device_status() == 8   # VD_ERR_DEVICE_BUDGET (sequence 0)
    assert cache.len.tolist() == [N + 3, N]
    assert torch.equal(before_v[0].view(torch.int16), cache.v[0].view(torch.int16))
    cache.len.copy_(torch.tensor([N + 6, N], dtype=torch.int32))
    vd.vd_evict_block(cache, N, None, 0, oracle.L2, vd.VD_MU_RECOMPUTE, None, None, None)
    assert vd.vd_get_device_status() == 7   # VD_ERR_DEVICE_LEN (sequence 0)
    assert cache.len.tolist() == [N + 6, N]


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_head_dim_256(orc, var):
    """The widest head dim: 4 * capacity * 256 <= 64 KB leaves 64 rows."""
    d, cap, N, B = 256, 64, 40, 24
    cache = filled_cache(2, 1, 3, cap, d, [cap, N + 5], seed=81)
    evict_and_check(orc, cache, N, B, var, vd.VD_MU_RECOMPUTE)


def test_nan_row_is_reported_and_evicted_first(orc):
    """A NaN in one row makes its Norm score NaN (the Norm rule reads no
    mean, so the other rows keep finite scores): the event is still run, the
    status reports VD_ERR_NONFINITE, and that row is evicted before any
    other (NaN ranks lowest), as in the oracle."""
    d, n, N = 64, 100, 99
    cache = filled_cache(1, 1, 2, n, d, [n], seed=83)
    cache.v[0, 0, 0, 37, 5] = float("nan")
    kept = torch.full(cache.unit_shape() + (N,), -7, dtype=torch.int32, device="cuda")
    pre_v = bits(units_view(cache.v))
    vd.vd_evict_block(cache, N, None, 0, oracle.NORM, vd.VD_MU_RECOMPUTE, None, kept, None)
    assert vd.vd_get_device_status() == 4   # VD_ERR_NONFINITE
    kh = kept.view(2, N).cpu().numpy()
    assert 37 not in kh[0].tolist()          # the NaN row went
    # unit 1 has no NaN: it evicts its lowest score, as the oracle does
    s0 = orc.scores(pre_v[0, :n], oracle.NORM)
    assert np.isnan(s0[37]) and np.array_equal(kh[0], orc.select_top_n(s0, N))
    s1 = orc.scores(pre_v[1, :n], oracle.NORM)
    assert np.array_equal(kh[1], orc.select_top_n(s1, N))
