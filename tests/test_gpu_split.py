"""Split launches: the units of one call run as two launches on the stream,
the first (units [0, s)) one CTA per unit, the second (units [s, U)) a
cluster of c CTAs per unit, started as a programmatic dependent of the
first so that its CTAs take the slots the first leaves free.

A unit's arithmetic depends only on the number of CTAs that process it, so
every output of a split call must equal, unit by unit, the same call run
unsplit at cluster size 1 (units below s) and at cluster size c (the
rest): scores, kept slots, sigma, compacted K and V, the running sum,
positions and lengths, bit for bit.  The automatic split (prefill-size
hole-fill and score-only launches with more units than SMs) is checked
against the fp64 oracle as well.  Needs a GB300."""
from __future__ import annotations

import contextlib
import os
import zlib

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from test_gpu_holefill import run_event
from vd_gpu import bits, check_scores, new_cache, units_view

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
def env(**kw):
    old = {k: os.environ.get(k) for k in kw}
    for k, v in kw.items():
        if v is None:
            os.environ.pop(k, None)
        else:
            os.environ[k] = str(v)
    try:
        yield
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def make(n_seq, L, H, cap, d, lens, seed, gen="student_t", B=0):
    cache = new_cache(n_seq, L, H, cap, d)
    st = wl.TokenStream(gen, cache.units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    us = cache.unit_shape()
    kn = vn = None
    if B:
        k, v = st.next(B)
        kn, vn = k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()
    return cache, kn, vn


def snapshot(cache, outs):
    """Host copies of everything a call may write, per unit where per unit."""
    U = cache.units
    res = {"k": bits(units_view(cache.k)), "v": bits(units_view(cache.v)),
           "len": cache.len.cpu().numpy().copy()}
    for name, t in outs.items():
        if t is not None:
            a = t.cpu().numpy().copy()
            res[name] = a.reshape(U, -1) if a.size % U == 0 and name != "len" else a
    return res


def run_call(kind, cache0, kn, vn, var, mu, N, B, c, solo):
    """One call of `kind` on a copy of cache0 with cluster size c (and a
    forced split of `solo` units when solo > 0); returns its outputs."""
    cache = vd.Cache(cache0.k.clone(), cache0.v.clone(), cache0.len.clone())
    us, U, cap, d = cache.unit_shape(), cache.units, cache.capacity, cache.head_dim
    outs = {"kept": torch.full(us + (N,), -7, dtype=torch.int32, device="cuda"),
            "scores": torch.full(us + (cap,), float("nan"), device="cuda")}
    rs = None
    score_keys = kind.endswith("_k")
    if mu == vd.VD_MU_RUNNING:
        rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
        vd.vd_running_sum_init_ex(cache, score_keys, rs)
        outs["rs"] = rs
    pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(U).view(us + (cap,)).contiguous()
    lens = cache.len.clone()
    with env(VD_CLUSTER_SIZE=c, VD_SOLO_UNITS=solo if solo else None):
        if kind == "holefill":
            pn = (lens - B).clone()
            vd.vd_evict_block_holefill(cache, N, pos, pn, None, B, var, mu, rs, outs["kept"],
                                       outs["scores"])
            outs["pos"] = pos
        elif kind == "holefill_fused":
            pn = lens.clone()
            vd.vd_append_evict_block(cache, kn, vn, B, N, None, var, mu, rs, outs["kept"],
                                     outs["scores"], pos=pos, pos_first_new=pn)
            outs["pos"] = pos
        elif kind == "ordered_fused":
            vd.vd_append_evict_block(cache, kn, vn, B, N, None, var, mu, rs, outs["kept"],
                                     outs["scores"])
        elif kind == "decode":
            outs["ev"] = torch.full(us, -7, dtype=torch.int32, device="cuda")
            vd.vd_evict_decode(cache, N, None, var, mu, rs, outs["ev"], outs["kept"],
                               outs["scores"])
        elif kind in ("options", "options_k"):
            g = torch.Generator(device="cuda").manual_seed(3)
            attn = torch.rand(us + (cap,), generator=g, device="cuda") * 0.9
            outs["sigma"] = torch.full(us, float("nan"), device="cuda")
            vd.vd_evict_block_ex(cache, N, None, B, var, mu, rs, score_keys, attn, outs["kept"],
                                 outs["scores"], outs["sigma"] if var == oracle.L2 else None)
        elif kind in ("score", "score_k"):
            outs.pop("kept")
            if var == oracle.L2:
                outs["sigma"] = torch.full(us, float("nan"), device="cuda")
            vd.vd_score_ex(cache, var, score_keys, outs["scores"], outs.get("sigma"), mu=mu,
                           running_sum=rs)
        else:
            raise ValueError(kind)
    assert vd.vd_get_device_status() == 0
    torch.cuda.synchronize()
    return snapshot(cache, outs)


def assert_unitwise(split, ref1, refc, solo, n_seq):
    for name in split:
        a = split[name]
        if name == "len":
            assert np.array_equal(a, ref1[name]) and np.array_equal(a, refc[name]), name
            continue
        lo = a[:solo].view(np.uint8) if a.dtype.kind == "f" else a[:solo]
        hi = a[solo:].view(np.uint8) if a.dtype.kind == "f" else a[solo:]
        r1, rc = ref1[name][:solo], refc[name][solo:]
        if a.dtype.kind == "f":
            r1, rc = r1.view(np.uint8), rc.view(np.uint8)
        assert np.array_equal(lo, r1), f"{name}: first part differs from the one-CTA launch"
        assert np.array_equal(hi, rc), f"{name}: second part differs from the cluster launch"


CASES = [
    # kind, head dim, N, B, cluster size c of the second part, units of the first part
    ("holefill", 128, 300, 64, 4, 3),
    ("holefill_fused", 256, 256, 64, 4, 5),
    ("holefill_fused", 64, 200, 40, 2, 7),
    ("ordered_fused", 128, 300, 64, 8, 2),
    ("decode", 128, 400, 1, 4, 6),
    ("options", 128, 300, 64, 2, 4),
    ("options_k", 256, 260, 60, 4, 4),
    ("score", 128, 300, 0, 4, 5),
    ("score_k", 64, 300, 0, 2, 3),
]


@pytest.mark.parametrize("mu", [vd.VD_MU_RECOMPUTE, vd.VD_MU_RUNNING], ids=["recompute", "running"])
@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
@pytest.mark.parametrize("case", CASES, ids=[f"{c[0]}-d{c[1]}-c{c[4]}-s{c[5]}" for c in CASES])
def test_split_equals_unsplit_unitwise(case, var, mu):
    kind, d, N, B, c, solo = case
    n_seq, L, H = 3, 2, 2                    # 12 units, 4 per sequence
    fused = kind.endswith("fused")
    cap = N + max(B, 1)
    if kind.startswith("score"):
        lens = [cap, cap - 7, cap // 2]
    elif fused:
        lens = [N, N - 3, N - B - 5]         # the third does not evict
    else:
        lens = [cap, N + 1 if kind == "decode" else N + 3, N - 9]
    cache, kn, vn = make(n_seq, L, H, cap, d, lens, seed=zlib.crc32(repr(case).encode()) % 1000, B=B if fused else 0)
    split = run_call(kind, cache, kn, vn, var, mu, N, B, c, solo)
    ref1 = run_call(kind, cache, kn, vn, var, mu, N, B, 1, 0)
    refc = run_call(kind, cache, kn, vn, var, mu, N, B, c, 0)
    assert_unitwise(split, ref1, refc, solo, n_seq)


@pytest.mark.parametrize("var", VARS, ids=VAR_IDS)
def test_automatic_split_holefill_against_oracle(orc, var):
    """More units than SMs, one wave at one CTA per unit: the automatic plan
    splits the launch.  Every unit checked against the oracle through token
    positions, with the running mean."""
    props = torch.cuda.get_device_properties(0)
    sms = props.multi_processor_count
    d, N, B = 128, 256, 64
    n_seq, L, H = 1, sms + 13, 1             # units_per_seq > SMs, not a multiple of it
    cap = N + B
    cache, _, _ = make(n_seq, L, H, cap, d, [cap], seed=77, gen="gauss_outlier")
    U = cache.units
    pos = torch.arange(cap, dtype=torch.int32, device="cuda").repeat(U).view(
        cache.unit_shape() + (cap,)).contiguous()
    rs = torch.zeros(cache.unit_shape() + (d,), dtype=torch.float64, device="cuda")
    cache.len.fill_(N)                       # the running sum of the rows before the block
    vd.vd_running_sum_init(cache, rs)
    cache.len.fill_(cap)
    with env(VD_CLUSTER_SIZE=None, VD_SOLO_UNITS=None, VD_SPLIT_LAUNCH=None):
        run_event(orc, var, cache, pos, torch.tensor([N], dtype=torch.int32, device="cuda"),
                  N, B, vd.VD_MU_RUNNING, rs)
    ref = torch.zeros_like(rs)
    vd.vd_running_sum_init(cache, ref)
    assert torch.max(torch.abs(ref - rs)).item() <= 1e-9


@pytest.mark.parametrize("var", [oracle.L2, oracle.NORM], ids=["l2", "norm"])
def test_automatic_split_score_pass_against_oracle(orc, var):
    """Score-only launch with more units than SMs (bulk-copy ring): scores
    of every unit within the parity tolerance of the oracle."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    d, cap = 256, 700
    cache, _, _ = make(1, sms + 21, 1, cap, d, [cap - 3], seed=11)
    U = cache.units
    sc = torch.full(cache.unit_shape() + (cap,), float("nan"), device="cuda")
    with env(VD_CLUSTER_SIZE=None, VD_SOLO_UNITS=None, VD_SPLIT_LAUNCH=None):
        vd.vd_score(cache, var, sc)
    assert vd.vd_get_device_status() == 0
    v = bits(units_view(cache.v))
    s = sc.view(U, cap).cpu().numpy()
    n = cap - 3
    for u in range(U):
        check_scores(orc, var, v[u][:n], s[u][:n])
