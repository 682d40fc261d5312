"""Seeded random sweep of the fused entry points against the fp64 oracle.

Each case draws a shape (sequences, layers, KV heads, a head dim that is a
multiple of 8 up to 256), a budget N, a block size B (1 for decode), ragged
lengths at or below N, a scoring rule, a mean mode, a layout and a cluster
size (with it, in 40 % of the cases, a split launch: the first units one
CTA each, the rest on clusters of that size), per-sequence budgets or not, fills the cache from the workload
generators, and runs two events through vd_append_evict_block /
vd_append_evict_decode (or, in some cases, the two-call form: vd_append,
then the eviction of that layout).  Every unit of every
event is checked like the rest of the parity suite: scores within 1e-5
relative of the oracle's (plus the fp32 rounding floor), the kept set of
Eq. (eviction) outside near ties, the compacted K and V rows bit for bit, the
new length, and the running sum against a from-scratch sum.  Needs a GB300.
"""
from __future__ import annotations

import os

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from test_gpu_holefill import check_holefill_event
from vd_gpu import bits, check_event, new_cache, units_view

pytestmark = pytest.mark.gpu
HEAD_DIMS = [8, 16, 24, 40, 64, 72, 128, 136, 200, 256]
# case counts (VD_FUZZ_CASES / VD_FUZZ_MEDIUM / VD_FUZZ_EX widen a run)
N_CASES = int(os.environ.get("VD_FUZZ_CASES", "48"))
N_MEDIUM = int(os.environ.get("VD_FUZZ_MEDIUM", "8"))  # budgets of 1000-6000 tokens


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def draw_case(i, medium=False):
    r = np.random.default_rng(7919 * (i + 1) + (104729 if medium else 0))
    d = int(r.choice([64, 128, 256] if medium else HEAD_DIMS))
    decode = bool(r.random() < 0.35)
    N = int(r.integers(1000, 6001)) if medium else int(r.integers(1, 401))
    B = 1 if decode else int(r.integers(1, 513 if medium else 97))
    n_seq, L, H = int(r.integers(1, 4)), int(r.integers(1, 3)), int(r.integers(1, 4))
    budgets = [int(r.integers(1, N + 1)) for _ in range(n_seq)] if r.random() < 0.3 else None
    lens = [int(r.integers(max(0, Nb - 3 * B), Nb + 1))
            for Nb in (budgets if budgets else [N] * n_seq)]
    allowed = [c for c in (1, 2, 4, 8, 16) if (2 * (d // 8)) % c == 0]
    return dict(d=d, decode=decode, N=N, B=B, n_seq=n_seq, L=L, H=H, lens=lens,
                budgets=budgets, two_call=bool(r.random() < 0.2),
                cap=N + B + int(r.integers(0, 17)),
                var=int(r.integers(0, 3)), mu=int(r.integers(0, 2)),
                holefill=bool(r.random() < 0.4),
                cluster=int(r.choice(allowed)) if r.random() < 0.5 else 0,
                gen=str(r.choice(["gauss_outlier", "student_t"])), seed=int(r.integers(1, 1 << 30)),
                split=float(r.random()))


def force_split(c, monkeypatch):
    """With a forced cluster size, 40 % of the cases also force a split
    launch: the first s units (1 <= s < U) one CTA each, the rest on
    clusters of the forced size."""
    U = c["n_seq"] * c["L"] * c["H"]
    if c["cluster"] and U >= 2 and c["split"] < 0.4:
        s = 1 + min(U - 2, int(c["split"] / 0.4 * (U - 1)))
        monkeypatch.setenv("VD_SOLO_UNITS", str(s))


@pytest.mark.parametrize("case", [(i, False) for i in range(N_CASES)] +
                         [(i, True) for i in range(N_MEDIUM)],
                         ids=[f"small{i}" for i in range(N_CASES)] +
                         [f"medium{i}" for i in range(N_MEDIUM)])
def test_fused_random_shapes(orc, case, monkeypatch):
    c = draw_case(*case)
    if c["cluster"]:
        monkeypatch.setenv("VD_CLUSTER_SIZE", str(c["cluster"]))
    force_split(c, monkeypatch)
    d, N, B, cap = c["d"], c["N"], c["B"], c["cap"]
    cache = new_cache(c["n_seq"], c["L"], c["H"], cap, d)
    U, us, per_seq = cache.units, cache.unit_shape(), c["L"] * c["H"]
    st = wl.TokenStream(c["gen"], U, d, device="cuda", seed=c["seed"])
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(c["lens"], dtype=torch.int32))
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    if c["mu"] == vd.VD_MU_RUNNING:
        vd.vd_running_sum_init(cache, rs)
    pos = pos_new = None
    if c["holefill"]:
        pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(U).view(us + (cap,))
        pos = pos.contiguous()
    N_dev = (torch.tensor(c["budgets"], dtype=torch.int32, device="cuda")
             if c["budgets"] else None)
    Ns = c["budgets"] if c["budgets"] else [N] * c["n_seq"]
    for event in range(2):
        lens = cache.len.cpu().numpy().copy()
        pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
        pre_pos = pos.view(U, cap).cpu().numpy().copy() if pos is not None else None
        k_new, v_new = st.next(B)
        k_new, v_new = k_new.view(us + (B, d)).contiguous(), v_new.view(us + (B, d)).contiguous()
        kn, vn = bits(k_new.view(U, B, d)), bits(v_new.view(U, B, d))
        if pos is not None:
            pos_new = torch.full((c["n_seq"],), cap + 1000 * (event + 1), dtype=torch.int32,
                                 device="cuda")
        kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
        scores = torch.full(us + (cap,), float("nan"), device="cuda")
        evicted = torch.full(us, -7, dtype=torch.int32, device="cuda")
        rs_arg = rs if c["mu"] == vd.VD_MU_RUNNING else None
        if c["two_call"]:
            vd.vd_append(cache, k_new, v_new, B)
            if c["decode"] and pos is not None:
                vd.vd_evict_decode_holefill(cache, N, pos, pos_new, N_dev, c["var"], c["mu"],
                                            rs_arg, evicted, kept, scores)
            elif c["decode"]:
                vd.vd_evict_decode(cache, N, N_dev, c["var"], c["mu"], rs_arg, evicted, kept,
                                   scores)
            elif pos is not None:
                vd.vd_evict_block_holefill(cache, N, pos, pos_new, N_dev, B, c["var"], c["mu"],
                                           rs_arg, kept, scores)
            else:
                vd.vd_evict_block(cache, N, N_dev, B, c["var"], c["mu"], rs_arg, kept, scores)
        elif c["decode"]:
            vd.vd_append_evict_decode(cache, k_new, v_new, N, N_dev, c["var"], c["mu"], rs_arg,
                                      evicted, kept, scores, pos=pos, pos_first_new=pos_new)
        else:
            vd.vd_append_evict_block(cache, k_new, v_new, B, N, N_dev, c["var"], c["mu"], rs_arg,
                                     kept, scores, pos=pos, pos_first_new=pos_new)
        assert vd.vd_get_device_status() == 0, c
        post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
        new_lens = cache.len.cpu().numpy()
        kh, sh = kept.view(U, N).cpu().numpy(), scores.view(U, cap).cpu().numpy()
        post_pos = pos.view(U, cap).cpu().numpy() if pos is not None else None
        for u in range(U):
            s = u // per_seq
            len0 = int(lens[s])  # read before the call: the pre-append length
            n, Nb = len0 + B, Ns[s]
            assert new_lens[s] == min(n, Nb), (c, event, u)
            # the rows the event saw: the cache's len0 rows, then the new ones
            ek = np.concatenate([pre_k[u, :len0], kn[u]])
            ev = np.concatenate([pre_v[u, :len0], vn[u]])
            if pos is None:
                check_event(orc, c["var"], ek, ev, post_k[u], post_v[u], n, Nb,
                            kh[u] if n > Nb else None, sh[u] if n > Nb else None)
            else:
                ep = np.concatenate([pre_pos[u, :len0], int(pos_new[s]) + np.arange(B)])
                check_holefill_event(orc, c["var"], ek, ev, ep.astype(np.int32), post_k[u],
                                     post_v[u], post_pos[u], n, Nb, kh[u] if n > Nb else None,
                                     sh[u] if n > Nb else None)
        if c["mu"] == vd.VD_MU_RUNNING:
            ref = torch.zeros_like(rs)
            vd.vd_running_sum_init(cache, ref)
            scale = units_view(cache.v).float().abs().sum(dim=1).max().item() + 1.0
            assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale, (c, event)


N_EX = int(os.environ.get("VD_FUZZ_EX", "24"))  # the scoring options of vd_evict_block_ex


def draw_ex(i):
    r = np.random.default_rng(31337 * (i + 1))
    d = int(r.choice(HEAD_DIMS))
    N, B = int(r.integers(1, 401)), int(r.integers(1, 97))
    n_seq, L, H = int(r.integers(1, 4)), int(r.integers(1, 3)), int(r.integers(1, 4))
    var = int(r.integers(0, 3))
    allowed = [c for c in (1, 2, 4, 8, 16) if (2 * (d // 8)) % c == 0]
    return dict(d=d, N=N, B=B, n_seq=n_seq, L=L, H=H,
                lens=[int(r.integers(max(0, N - 2 * B), N + 1)) for _ in range(n_seq)],
                cap=N + B + int(r.integers(0, 17)), var=var, keys=bool(r.random() < 0.5),
                weighted=bool(r.random() < 0.4), disp=var == 0 and bool(r.random() < 0.5),
                mu=int(r.integers(0, 2)),
                cluster=int(r.choice(allowed)) if r.random() < 0.5 else 0,
                gen=str(r.choice(["gauss_outlier", "student_t"])), seed=int(r.integers(1, 1 << 30)),
                fused=bool(r.random() < 0.5), split=float(r.random()))


@pytest.mark.parametrize("case", range(N_EX))
def test_ex_random_options(orc, case, monkeypatch):
    """One block event through vd_evict_block_ex (after vd_append) or
    vd_append_evict_block_ex with random scoring options:
    scores of the scored tensor (K for the key-side rule) within the parity
    tolerance (weighted: scaled by the factor a/(1 - a), App. A), the kept
    set outside near ties, bit-exact gathers, sigma of the plain L2 scores
    for the units that evicted, and the running sum of the scored tensor."""
    import test_gpu_extensions as tx
    from vd_gpu import score_tolerance, weighted_tolerance
    tx._ORC = orc
    c = draw_ex(case)
    if c["cluster"]:
        monkeypatch.setenv("VD_CLUSTER_SIZE", str(c["cluster"]))
    force_split(c, monkeypatch)
    d, N, B, cap, var = c["d"], c["N"], c["B"], c["cap"], c["var"]
    cache = new_cache(c["n_seq"], c["L"], c["H"], cap, d)
    U, us, per_seq = cache.units, cache.unit_shape(), c["L"] * c["H"]
    st = wl.TokenStream(c["gen"], U, d, device="cuda", seed=c["seed"])
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(c["lens"], dtype=torch.int32))
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    running = c["mu"] == vd.VD_MU_RUNNING
    if running:
        vd.vd_running_sum_init_ex(cache, c["keys"], rs)
    k_new, v_new = st.next(B)
    k_new, v_new = k_new.view(us + (B, d)).contiguous(), v_new.view(us + (B, d)).contiguous()
    if c["fused"]:
        # the event's rows: the cached ones, then the new ones at slots len ..
        lens = cache.len.cpu().numpy().copy() + B
        pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
        kn, vn = bits(k_new.view(U, B, d)), bits(v_new.view(U, B, d))
        for u in range(U):
            n0 = int(lens[u // per_seq]) - B
            pre_k[u, n0:n0 + B], pre_v[u, n0:n0 + B] = kn[u], vn[u]
    else:
        vd.vd_append(cache, k_new, v_new, B)
        lens = cache.len.cpu().numpy().copy()
        pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    attn = None
    if c["weighted"]:
        g = torch.Generator(device="cuda").manual_seed(c["seed"] % 100003)
        attn = torch.rand(us + (cap,), generator=g, device="cuda") * 0.9
        attn[..., ::17] = 0.0
    kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
    scores = torch.full(us + (cap,), float("nan"), device="cuda")
    sigma = torch.full(us, -1.0, device="cuda") if c["disp"] else None
    if c["fused"]:
        vd.vd_append_evict_block_ex(cache, k_new, v_new, B, N, None, var, c["mu"],
                                    rs if running else None, c["keys"], attn, kept, scores, sigma)
    else:
        vd.vd_evict_block_ex(cache, N, None, B, var, c["mu"], rs if running else None,
                             c["keys"], attn, kept, scores, sigma)
    assert vd.vd_get_device_status() == 0, c
    post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    kh, sh = kept.view(U, N).cpu().numpy(), scores.view(U, cap).cpu().numpy()
    a_h = attn.view(U, cap).cpu().numpy().astype(np.float64) if attn is not None else None
    sg = sigma.view(U).cpu().numpy() if sigma is not None else None
    for u in range(U):
        n = int(lens[u // per_seq])
        src = pre_k[u, :n] if c["keys"] else pre_v[u, :n]
        if n <= N:
            assert np.array_equal(post_k[u, :n], pre_k[u, :n])
            assert np.array_equal(post_v[u, :n], pre_v[u, :n])
            if sg is not None:
                assert sg[u] == -1.0, (c, u)
            continue
        if a_h is None:
            s_ora = orc.scores(src, var)
            tol = score_tolerance(var, s_ora, src, orc.mean(src))
        else:
            s_ora = orc.scores_weighted(src, a_h[u, :n], var)
            f = a_h[u, :n] / (1.0 - a_h[u, :n])
            tol = weighted_tolerance(var, s_ora, orc.scores(src, var), src, orc.mean(src), f)
        tx.check_scored_event(s_ora, tol, pre_k[u], pre_v[u], post_k[u], post_v[u], n, N, kh[u],
                              sh[u], var, ("_k" if c["keys"] else "") + ("_w" if a_h is not None else ""))
        if sg is not None:
            want = orc.dispersion(src)
            assert abs(sg[u] - want) <= 1e-5 * want + 1e-6, (c, u, sg[u], want)
    if running:
        ref = torch.zeros_like(rs)
        vd.vd_running_sum_init_ex(cache, c["keys"], ref)
        t = units_view(cache.k if c["keys"] else cache.v)
        scale = t.float().abs().sum(dim=1).max().item() + 1.0
        assert torch.max(torch.abs(ref - rs)).item() <= 1e-12 * scale, c
