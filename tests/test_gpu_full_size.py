"""Parity at the five workloads' full sizes, in the launch configuration the
benchmark times (its workload classes and the library's own cluster choice):
sampled units against the fp64 oracle, step-locked, plus properties checked
on every unit (length, slot lists, bit-exact gathers, running sum against a
from-scratch recompute).  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import bench
import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import bits, check_event, units_view

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    torch.cuda.empty_cache()


def sample_units(U, k, seed):
    rng = np.random.default_rng(seed)
    return sorted(rng.choice(U, size=min(k, U), replace=False).tolist())


def snapshot(cache, units):
    it = torch.tensor(units, device=DEV, dtype=torch.long)
    return bits(units_view(cache.k)[it]), bits(units_view(cache.v)[it])


def snapshot_step(w, units):
    """Pre-eviction rows of the benchmark's next step: the cache's rows and,
    where the step appends inside the eviction call (vd_append_evict_block),
    the staged block after them.  Returns (k, v, n)."""
    k, v = snapshot(w.cache, units)
    n0 = int(w.cache.len[0])
    if not getattr(w, "fused", False):
        return k, v, n0
    it = torch.tensor(units, device=DEV, dtype=torch.long)
    pk, pv = w.pending
    k, v = k.copy(), v.copy()
    k[:, n0:n0 + w.B] = bits(pk.view(w.U, w.B, w.d)[it])
    v[:, n0:n0 + w.B] = bits(pv.view(w.U, w.B, w.d)[it])
    return k, v, n0 + w.B


def check_sampled(orc, var, cache, units, pre, n_of, N_of, kept, scores):
    post = snapshot(cache, units)
    U = cache.units
    per_seq = cache.n_layer * cache.n_kv_head
    kept_h = kept.view(U, -1).cpu().numpy()
    sc_h = scores.view(U, -1).cpu().numpy() if scores is not None else None
    lens = cache.len.cpu().numpy()
    for i, u in enumerate(units):
        s = u // per_seq
        check_event(orc, var, pre[0][i], pre[1][i], post[0][i], post[1][i], int(n_of(s)),
                    int(N_of(s)), kept_gpu=kept_h[u],
                    scores_gpu=None if sc_h is None else sc_h[u], new_len=int(lens[s]))


def check_all_units_gather(pre_k, pre_v, cache, kept, N, units_idx):
    """Bit-exact gather on every listed unit: post[r] = pre[kept[r]]."""
    it = units_idx
    post_k = units_view(cache.k)[it][:, :N]
    post_v = units_view(cache.v)[it][:, :N]
    kk = kept.view(cache.units, -1)[it][:, :N].long()
    assert torch.all(kk[:, 1:] > kk[:, :-1]), "kept slots must be strictly ascending"
    idx = kk.unsqueeze(-1).expand(-1, -1, cache.head_dim)
    assert torch.equal(torch.gather(pre_v, 1, idx).view(torch.int16), post_v.view(torch.int16))
    assert torch.equal(torch.gather(pre_k, 1, idx).view(torch.int16), post_k.view(torch.int16))


def check_running_sum(cache, rs):
    """The running sum after many events equals a from-scratch sum of the
    cached rows within 1e-12 of sum |v| (bounded here by n * max |v|)."""
    ref = torch.zeros_like(rs)
    vd.vd_running_sum_init(cache, ref)
    assert vd.vd_get_device_status() == 0
    n = int(cache.len.max())
    scale = n * units_view(cache.v)[:, :n].abs().max().float().item()
    err = torch.max(torch.abs(ref - rs)).item()
    assert err <= 1e-12 * scale, (err, scale)


# ---------------------------------------------------------------------------
# prefill configurations: the whole prompt, block by block, from an empty cache
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["tiny_prefill", "prefill_gqa8b", "prefill_wide"])
def test_full_prompt_block_processing(orc, name):
    _, cfg = wl.config(name)
    d, N, B, T = cfg["head_dim"], cfg["N"], cfg["B"], cfg["T"]
    cache = vd.Cache.empty(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], N + B, d, device=DEV)
    U = cache.units
    us = cache.unit_shape()
    st = wl.stream_for(cfg, device="cuda")
    rs = torch.zeros(us + (d,), dtype=torch.float64, device=DEV)
    kept = torch.empty(us + (N,), dtype=torch.int32, device=DEV)
    scores = torch.empty(us + (N + B,), dtype=torch.float32, device=DEV)
    n_blocks = T // B
    first_evict = N // B                 # block index at which len first exceeds N
    check_at = {first_evict, n_blocks // 2, n_blocks - 1}
    units = sample_units(U, 6, cfg["index"])
    all_units = torch.arange(0, U, max(1, U // 64), device=DEV)
    for blk in range(n_blocks):
        k, v = st.next(B)
        vd.vd_append(cache, k.view(us + (B, d)), v.view(us + (B, d)), B)
        if blk in check_at:
            n = int(cache.len[0])
            pre = snapshot(cache, units)
            pre_k = units_view(cache.k)[all_units].clone()
            pre_v = units_view(cache.v)[all_units].clone()
            vd.vd_evict_block(cache, N, None, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, kept, scores)
            assert vd.vd_get_device_status() == 0
            check_sampled(orc, oracle.L2, cache, units, pre, lambda s: n, lambda s: N, kept, scores)
            if n > N:
                check_all_units_gather(pre_k, pre_v, cache, kept, N, all_units)
            check_running_sum(cache, rs)
        else:
            vd.vd_evict_block(cache, N, None, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, None, None)
    assert vd.vd_get_device_status() == 0
    assert int(cache.len[0]) == N
    check_running_sum(cache, rs)


@pytest.mark.parametrize("var", [oracle.L2, oracle.DIR, oracle.NORM], ids=["l2", "dir", "norm"])
@pytest.mark.parametrize("mu", ["running", "recompute"])
def test_prefill_wide_steady_state_as_benchmarked(orc, var, mu):
    """The benchmark's own steady-state prefill_wide event (336 units,
    4352 -> 4096, d = 256), sampled units against the oracle."""
    _, cfg = wl.config("prefill_wide")
    mu_c = vd.VD_MU_RUNNING if mu == "running" else vd.VD_MU_RECOMPUTE
    w = bench.Prefill("prefill_wide", cfg, DEV, wl.BASE_SEED + 2, mu_c, var)
    units = sample_units(w.U, 4, 7 + var)
    kept = torch.empty(w.cache.unit_shape() + (w.N,), dtype=torch.int32, device=DEV)
    scores = torch.empty(w.cache.unit_shape() + (w.cap,), dtype=torch.float32, device=DEV)
    assert w.fused                      # the benchmark's step: one vd_append_evict_block call
    for step in range(3):
        w.append_next()
        pk, pv, n = snapshot_step(w, units)
        assert n == w.N + w.B
        w.evict(kept, scores)
        assert vd.vd_get_device_status() == 0
        check_sampled(orc, var, w.cache, units, (pk, pv), lambda s: n, lambda s: w.N, kept,
                      scores)
    if mu == "running":
        check_running_sum(w.cache, w.rs)
    del w
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------
# batched decode: 64 x 32 x 8 units at N = 4096, 1024 steps, running mean
# checked against recompute every 64 steps
# ---------------------------------------------------------------------------
def test_decode_batched_1024_steps(orc):
    _, cfg = wl.config("decode_batched")
    w = bench.Decode("decode_batched", cfg, DEV, wl.BASE_SEED + 3, vd.VD_MU_RUNNING,
                     vd.VD_SCORE_L2)
    U, d, N = w.U, w.d, w.N
    us = w.cache.unit_shape()
    st = wl.stream_for(cfg, device="cuda", seed=wl.BASE_SEED + 300)
    evicted = torch.empty(us, dtype=torch.int32, device=DEV)
    kept = torch.empty(us + (N,), dtype=torch.int32, device=DEV)
    scores = torch.empty(us + (N + 1,), dtype=torch.float32, device=DEV)
    units = sample_units(U, 8, 33)
    sub = torch.arange(0, U, 16, device=DEV)           # 1024 units for whole-unit checks
    for step in range(cfg["steps"]):
        k, v = st.next(1)
        w.append_next(k.view(us + (1, d)), v.view(us + (1, d)))
        if step in (0, 511, 1023):
            assert w.fused                  # the benchmark's step: one vd_append_evict_decode call
            pk, pv, n = snapshot_step(w, units)
            assert n == N + 1
            pre = (pk, pv)
            pre_k = units_view(w.cache.k)[sub].clone()
            pre_v = units_view(w.cache.v)[sub].clone()
            pre_k[:, N] = w.pending[0].view(U, d)[sub]     # the staged token at slot N
            pre_v[:, N] = w.pending[1].view(U, d)[sub]
            w.evict(evicted, kept, scores)
            assert vd.vd_get_device_status() == 0
            check_sampled(orc, oracle.L2, w.cache, units, pre, lambda s: N + 1, lambda s: N, kept,
                          scores)
            check_all_units_gather(pre_k, pre_v, w.cache, kept, N, sub)
            ev = evicted.view(U)
            assert torch.all((ev >= 0) & (ev <= N))
            # the evicted slot is the one missing from the kept list
            kk = kept.view(U, N)[sub].long()
            missing = torch.where((kk != torch.arange(N, device=DEV)).any(dim=1),
                                  (kk != torch.arange(N, device=DEV)).int().argmax(dim=1),
                                  torch.full((sub.numel(),), N, device=DEV))
            assert torch.equal(missing.int(), ev[sub])
        else:
            w.evict(evicted)
        if step % cfg["check_every"] == cfg["check_every"] - 1:
            assert vd.vd_get_device_status() == 0
            check_running_sum(w.cache, w.rs)
    assert torch.all(w.cache.len == N)
    del w
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------
# ratio budget: 16 x 28 x 4 units, prompt 512 in blocks of 128, then 16384
# decode steps with N_t = floor(L_t / 4) per sequence
# ---------------------------------------------------------------------------
def test_ratio_budget_full_generation(orc):
    _, cfg = wl.config("ratio_budget")
    d, B, P, G = cfg["head_dim"], cfg["B"], cfg["prompt"], cfg["gen_tokens"]
    N_max = wl.budget_at(cfg, P + G)
    cache = vd.Cache.empty(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], N_max + 1 + B, d,
                           device=DEV)
    U = cache.units
    us = cache.unit_shape()
    st = wl.stream_for(cfg, device="cuda")
    rs = torch.zeros(us + (d,), dtype=torch.float64, device=DEV)
    N_dev = torch.empty(cfg["n_seq"], dtype=torch.int32, device=DEV)
    kept = torch.empty(us + (N_max,), dtype=torch.int32, device=DEV)
    scores = torch.empty(us + (cache.capacity,), dtype=torch.float32, device=DEV)
    evicted = torch.empty(us, dtype=torch.int32, device=DEV)
    units = sample_units(U, 6, 44)
    total = 0
    for _ in range(P // B):                      # prompt, block prompt processing
        k, v = st.next(B)
        vd.vd_append(cache, k.view(us + (B, d)), v.view(us + (B, d)), B)
        total += B
        N_t = wl.budget_at(cfg, total)
        N_dev.fill_(N_t)
        pre = snapshot(cache, units)
        n = int(cache.len[0])
        vd.vd_evict_block(cache, N_max, N_dev, B, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, kept, scores)
        assert vd.vd_get_device_status() == 0
        check_sampled(orc, oracle.L2, cache, units, pre, lambda s: n, lambda s: N_t, kept, scores)
    assert int(cache.len[0]) == wl.budget_at(cfg, P)
    evictions = 0
    check_steps = {0, 1, 2, 3, G // 2 + 1, G - 1}
    for step in range(G):
        k, v = st.next(1)
        vd.vd_append(cache, k.view(us + (1, d)), v.view(us + (1, d)), 1)
        total += 1
        N_t = wl.budget_at(cfg, total)
        N_dev.fill_(N_t)
        if step in check_steps:
            n = int(cache.len[0])
            pre = snapshot(cache, units)
            vd.vd_evict_decode(cache, N_max, N_dev, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, evicted,
                               kept, scores)
            assert vd.vd_get_device_status() == 0
            check_sampled(orc, oracle.L2, cache, units, pre, lambda s: n, lambda s: N_t, kept,
                          scores)
            evictions += n > N_t
        else:
            vd.vd_evict_decode(cache, N_max, N_dev, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs, None,
                               None, None)
        if step % 4096 == 4095:
            check_running_sum(cache, rs)
    assert vd.vd_get_device_status() == 0
    assert int(cache.len[0]) == wl.budget_at(cfg, total) == N_max
    assert evictions >= 3
    check_running_sum(cache, rs)


# ---------------------------------------------------------------------------
# hole-fill layout at full size, in the benchmark's configuration
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", ["decode_batched", "prefill_wide"])
def test_holefill_full_size_as_benchmarked(orc, name):
    from test_gpu_holefill import check_holefill_event
    _, cfg = wl.config(name)
    cls = bench.Decode if cfg["kind"] == "decode" else bench.Prefill
    w = cls(name, cfg, DEV, wl.BASE_SEED + cfg["index"], vd.VD_MU_RUNNING, vd.VD_SCORE_L2,
            layout="holefill")
    U, cap, N = w.U, w.cap, w.N
    units = sample_units(U, 6, 55)
    it = torch.tensor(units, device=DEV, dtype=torch.long)
    per_seq = w.cache.n_layer * w.cache.n_kv_head
    kept = torch.empty(w.cache.unit_shape() + (N,), dtype=torch.int32, device=DEV)
    scores = torch.empty(w.cache.unit_shape() + (cap,), dtype=torch.float32, device=DEV)
    for step in range(4):
        w.append_next()
        pk, pv, n = snapshot_step(w, units)
        pre = (pk, pv)
        pre_pos = w.pos.view(U, cap)[it].cpu().numpy().copy()
        pn = w.pos_new_all[w.i - 1].cpu().numpy()
        for i, u in enumerate(units):
            pre_pos[i, n - w.B:n] = pn[u // per_seq] + np.arange(w.B)
        if cfg["kind"] == "decode":
            w.evict(None, kept, scores)
        else:
            w.evict(kept, scores)
        assert vd.vd_get_device_status() == 0
        post = snapshot(w.cache, units)
        post_pos = w.pos.view(U, cap)[it].cpu().numpy()
        kh = kept.view(U, N)[it].cpu().numpy()
        sh = scores.view(U, cap)[it].cpu().numpy()
        for i in range(len(units)):
            check_holefill_event(orc, oracle.L2, pre[0][i], pre[1][i], pre_pos[i], post[0][i],
                                 post[1][i], post_pos[i], n, N, kh[i], sh[i])
    check_running_sum(w.cache, w.rs)
    del w
    torch.cuda.empty_cache()
