"""Calls captured in a CUDA graph and replayed give the same bytes as the
same calls run eagerly: the block and decode evictions (whose length update
is a programmatic dependent launch), the hole-fill and score-only calls at
sizes that take the split launch (two launches, the second a programmatic
dependent of the first), and the short-cache kernel.  Needs a GB300."""
from __future__ import annotations

import pytest
import torch

import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import new_cache, units_view

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def make_state(n_seq, L, H, cap, d, lens, B, seed):
    cache = new_cache(n_seq, L, H, cap, d)
    st = wl.TokenStream("gauss_outlier", cache.units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    us = cache.unit_shape()
    k, v = st.next(max(B, 1))
    kn, vn = k.view(us + (max(B, 1), d)).contiguous(), v.view(us + (max(B, 1), d)).contiguous()
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    vd.vd_running_sum_init(cache, rs)
    pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(cache.units).view(
        us + (cap,)).contiguous()
    return {"k": cache.k, "v": cache.v, "len": cache.len, "rs": rs, "pos": pos, "kn": kn, "vn": vn,
            "kept": torch.full(us + (cap,), -7, dtype=torch.int32, device="cuda"),
            "scores": torch.full(us + (cap,), float("nan"), device="cuda"),
            "ev": torch.full(us, -7, dtype=torch.int32, device="cuda"),
            "sigma": torch.full(us, float("nan"), device="cuda")}


def clone(state):
    return {k: t.clone() for k, t in state.items()}


def call(kind, s, N, B):
    cache = vd.Cache(s["k"], s["v"], s["len"])
    us = cache.unit_shape()
    if kind == "ordered_block":
        vd.vd_append_evict_block(cache, s["kn"], s["vn"], B, N, None, vd.VD_SCORE_L2,
                                 vd.VD_MU_RUNNING, s["rs"], s["kept"].view(-1)[:cache.units * N]
                                 .view(us + (N,)), s["scores"])
    elif kind == "holefill_block":             # the new rows' positions start at len
        vd.vd_append_evict_block(cache, s["kn"], s["vn"], B, N, None, vd.VD_SCORE_L2,
                                 vd.VD_MU_RUNNING, s["rs"], s["kept"].view(-1)[:cache.units * N]
                                 .view(us + (N,)), s["scores"], pos=s["pos"],
                                 pos_first_new=s["pnew"])
    elif kind == "decode":
        vd.vd_append_evict_decode(cache, s["kn"][..., :1, :], s["vn"][..., :1, :], N, None,
                                  vd.VD_SCORE_L2, vd.VD_MU_RUNNING, s["rs"], s["ev"],
                                  s["kept"].view(-1)[:cache.units * N].view(us + (N,)),
                                  s["scores"])
    elif kind == "score":
        vd.vd_score_ex(cache, vd.VD_SCORE_L2, False, s["scores"], s["sigma"],
                       mu=vd.VD_MU_RUNNING, running_sum=s["rs"])
    else:
        raise ValueError(kind)


CASES = {
    # kind: (n_seq, layers, heads, capacity, d, lens, N, B)
    "ordered_block": (2, 3, 4, 640, 128, [512, 500], 512, 128),
    "holefill_block": (1, 20, 8, 320, 128, [256], 256, 64),        # 160 units: split launch
    "decode": (3, 4, 4, 1025, 128, [1024, 1024, 1000], 1024, 1),
    "score": (1, 21, 8, 700, 256, [697], 1, 0),                     # 168 units: split launch
    "short_cache": (1, 1, 2, 160, 64, [128], 128, 32),              # the short-cache kernel
}


@pytest.mark.parametrize("kind", list(CASES))
def test_graph_replay_matches_eager(kind):
    n_seq, L, H, cap, d, lens, N, B = CASES[kind]
    base = make_state(n_seq, L, H, cap, d, lens, B, seed=len(kind))
    base["pnew"] = base["len"].clone()
    how = "ordered_block" if kind == "short_cache" else kind
    eager = clone(base)
    call(how, eager, N, B)
    torch.cuda.synchronize()
    assert vd.vd_get_device_status() == 0
    # the plan for this shape is cached by the eager call; capture on static
    # buffers, put the initial state back, replay once
    static = clone(base)
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        warm = clone(base)
        call(how, warm, N, B)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call(how, static, N, B)
    for k, t in base.items():
        static[k].copy_(t)
    g.replay()
    torch.cuda.synchronize()
    assert vd.vd_get_device_status() == 0
    for k in eager:
        a, b = eager[k], static[k]
        if a.dtype.is_floating_point:
            a, b = a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8)
        assert torch.equal(a, b), f"{kind}: {k} differs between graph replay and eager"
