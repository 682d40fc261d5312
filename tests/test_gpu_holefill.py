"""Hole-fill layout (vd_evict_*_holefill) against the fp64 oracle.

The oracle evicts the logical cache: the pre-eviction rows sorted by token
position (which makes its lower-index tie-break the lower-position rule).
The GPU result must keep the same set of positions (outside near ties), hold
in every slot exactly the bytes of the pre-eviction row with that position,
leave every surviving row below N in its slot, and report in kept_idx_out
the pre-eviction slot of every slot's token.  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import bits, check_scores, near_tie_band, new_cache, units_view

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


def check_holefill_event(orc, var, pre_k, pre_v, pre_pos, post_k, post_v, post_pos, n, N,
                         kept_gpu, scores_gpu):
    pre_k, pre_v, pre_pos = pre_k[:n], pre_v[:n], pre_pos[:n]
    assert len(set(pre_pos.tolist())) == n, "positions must be distinct"
    if n <= N:
        assert np.array_equal(post_k[:n], pre_k) and np.array_equal(post_v[:n], pre_v)
        assert np.array_equal(post_pos[:n], pre_pos)
        return
    order = np.argsort(pre_pos, kind="stable")       # logical (position) order
    lv = pre_v[order]
    s_ora = orc.scores(lv, var)
    if scores_gpu is not None:
        check_scores(orc, var, lv, scores_gpu[:n][order])
    kept_logical = orc.select_top_n(s_ora, N)
    want = set(pre_pos[order][kept_logical].tolist())
    got_pos = post_pos[:N]
    assert len(set(got_pos.tolist())) == N, "surviving positions must be distinct"
    diff = want ^ set(got_pos.tolist())
    if diff:
        band = near_tie_band(s_ora, N)
        rank_of = {p: i for i, p in enumerate(pre_pos[order].tolist())}
        assert all(band[rank_of[p]] for p in diff), "kept positions differ outside near ties"
    slot_of = {p: j for j, p in enumerate(pre_pos.tolist())}
    for r in range(N):
        j = slot_of[int(got_pos[r])]
        assert np.array_equal(post_k[r], pre_k[j]) and np.array_equal(post_v[r], pre_v[j])
        if kept_gpu is not None:
            assert kept_gpu[r] == j
        if j < N:
            assert j == r, "a surviving row below N must not move"


def run_event(orc, var, cache, pos, pos_new, N, B, mu, rs, decode=False, N_dev=None):
    U, cap = cache.units, cache.capacity
    lens = cache.len.cpu().numpy().copy()
    per_seq = cache.n_layer * cache.n_kv_head
    pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    pre_pos = pos.view(U, cap).cpu().numpy().copy()
    pn = pos_new.cpu().numpy()
    for u in range(U):                      # the appended rows' positions
        s = u // per_seq
        first = lens[s] - B
        pre_pos[u, first:lens[s]] = pn[s] + np.arange(B)
    us = cache.unit_shape()
    kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
    scores = torch.full(us + (cap,), float("nan"), device="cuda")
    evicted = torch.full(us, -7, dtype=torch.int32, device="cuda")
    if decode:
        vd.vd_evict_decode_holefill(cache, N, pos, pos_new, N_dev, var, mu, rs, evicted, kept, scores)
    else:
        vd.vd_evict_block_holefill(cache, N, pos, pos_new, N_dev, B, var, mu, rs, kept, scores)
    assert vd.vd_get_device_status() == 0
    post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    post_pos = pos.view(U, cap).cpu().numpy()
    new_lens = cache.len.cpu().numpy()
    kept_h, sc_h = kept.view(U, N).cpu().numpy(), scores.view(U, cap).cpu().numpy()
    ev_h = evicted.view(U).cpu().numpy()
    Ns = N_dev.cpu().numpy() if N_dev is not None else np.full(cache.n_seq, N)
    for u in range(U):
        s = u // per_seq
        n, Nb = int(lens[s]), int(Ns[s])
        assert new_lens[s] == min(n, Nb)
        check_holefill_event(orc, var, pre_k[u], pre_v[u], pre_pos[u], post_k[u], post_v[u],
                             post_pos[u], n, Nb, kept_h[u] if n > Nb else None,
                             sc_h[u] if n > Nb else None)
        if decode:
            if n <= Nb:
                assert ev_h[u] == -1
            else:
                gone = set(pre_pos[u, :n].tolist()) - set(post_pos[u, :Nb].tolist())
                assert len(gone) == 1 and pre_pos[u, ev_h[u]] == gone.pop()


def fresh(n_seq, L, H, cap, d, lens, seed, **kw):
    cache = new_cache(n_seq, L, H, cap, d)
    st = wl.TokenStream(kw.pop("gen", "gauss_outlier"), cache.units, d, device="cuda", seed=seed, **kw)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(cache.units).view(
        cache.unit_shape() + (cap,)).contiguous()
    return cache, pos, st


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("cluster", [1, 2, 4])
def test_holefill_block_event(orc, var, cluster, monkeypatch):
    monkeypatch.setenv("VD_CLUSTER_SIZE", str(cluster))
    d, N, B = 128, 200, 56
    lens = [N + B, N + 3, N, 77]
    cache, pos, _ = fresh(4, 2, 2, N + B, d, lens, seed=cluster)
    pos_new = torch.tensor([x - B for x in lens], dtype=torch.int32, device="cuda")
    run_event(orc, var, cache, pos, pos_new, N, B, vd.VD_MU_RECOMPUTE, None)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_holefill_prefill_trajectory_running(orc, var):
    """Block prompt processing in the hole-fill layout with the running mean:
    every event step-locked through positions; the running sum tracks the
    cache."""
    _, cfg = wl.config("tiny_prefill")
    d, N, B, T = cfg["head_dim"], cfg["N"], cfg["B"], cfg["T"]
    cache = new_cache(1, 1, 2, N + B, d)
    us = cache.unit_shape()
    pos = torch.full(us + (N + B,), -1, dtype=torch.int32, device="cuda")
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    st = wl.stream_for(cfg)
    for blk in range(T // B):
        k, v = st.next(B)
        vd.vd_append(cache, k.view(us + (B, d)), v.view(us + (B, d)), B)
        pos_new = torch.tensor([blk * B], dtype=torch.int32, device="cuda")
        run_event(orc, var, cache, pos, pos_new, N, B, vd.VD_MU_RUNNING, rs)
    ref = torch.zeros_like(rs)
    vd.vd_running_sum_init(cache, ref)
    assert torch.max(torch.abs(ref - rs)).item() <= 1e-9


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_holefill_decode_steps(orc, var):
    d, N = 64, 96
    cache, pos, _ = fresh(3, 2, 2, N + 1, d, [N, N, N - 5], seed=31, gen="drift")
    rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(cache, rs)
    st = wl.TokenStream("drift", cache.units, d, seed=32)
    us = cache.unit_shape()
    t = torch.tensor([N, N, N - 5], dtype=torch.int32, device="cuda")   # next position
    for step in range(30):
        k, v = st.next(1)
        vd.vd_append(cache, k.view(us + (1, d)), v.view(us + (1, d)), 1)
        run_event(orc, var, cache, pos, t, N, 1, vd.VD_MU_RUNNING, rs, decode=True)
        t += 1
    ref = torch.zeros_like(rs)
    vd.vd_running_sum_init(cache, ref)
    assert torch.max(torch.abs(ref - rs)).item() <= 1e-9


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_holefill_ties_break_by_position(orc, var):
    """Exact ties (duplicates, small integers) with shuffled positions: the
    lower position must win, not the lower slot."""
    d, N, B = 64, 100, 40
    for kw in (dict(dup_fraction=0.4), dict(small_int=True)):
        cache, pos, _ = fresh(2, 1, 2, N + B, d, [N + B, N + B], seed=5, **kw)
        g = torch.Generator(device="cuda").manual_seed(9)
        perm = torch.stack([torch.randperm(N, generator=g, device="cuda")
                            for _ in range(cache.units)]).int()
        pos[..., :N] = perm.view(cache.unit_shape() + (N,)) * 3       # distinct, not slot order
        pos_new = torch.full((2,), 10_000, dtype=torch.int32, device="cuda")
        run_event(orc, var, cache, pos, pos_new, N, B, vd.VD_MU_RECOMPUTE, None)


def test_holefill_per_sequence_budgets(orc):
    d, cap = 128, 400
    lens = [400, 390, 120, 3]
    Ns = torch.tensor([300, 390, 60, 1], dtype=torch.int32, device="cuda")
    cache, pos, _ = fresh(4, 1, 3, cap, d, lens, seed=12)
    B = 0
    pos_new = torch.tensor(lens, dtype=torch.int32, device="cuda")
    run_event(orc, oracle.L2, cache, pos, pos_new, 390, B, vd.VD_MU_RECOMPUTE, None, N_dev=Ns)


def test_holefill_decode_moves_one_row():
    """A decode step in the hole-fill layout changes at most one slot below N
    and leaves every other row's bytes in place."""
    d, N = 128, 512
    cache, pos, _ = fresh(2, 4, 2, N + 1, d, [N + 1, N + 1], seed=40)
    before_k, before_v = cache.k.clone(), cache.v.clone()
    ev = torch.empty(cache.unit_shape(), dtype=torch.int32, device="cuda")
    vd.vd_evict_decode_holefill(cache, N, pos, torch.tensor([N, N], dtype=torch.int32,
                                                            device="cuda"),
                                evicted_out=ev)
    assert vd.vd_get_device_status() == 0
    changed = (cache.v[..., :N, :].view(torch.int16) != before_v[..., :N, :].view(torch.int16)).any(-1)
    assert int(changed.sum(-1).max()) <= 1
    evu = ev.view(-1)
    for u in range(cache.units):
        e = int(evu[u])
        vu = units_view(cache.v)[u]
        if e < N:
            assert torch.equal(vu[e].view(torch.int16), units_view(before_v)[u][N].view(torch.int16))
            assert int(pos.view(cache.units, -1)[u, e]) == N
