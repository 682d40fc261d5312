"""Size limits and empty inputs: block eviction at the largest capacity its
16-bit slot lists allow (65536) and one past it, decode beyond that limit
(it keeps no slot list), and sequences of length 0.  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import bits, check_event, new_cache, units_view

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


def filled(n_seq, cap, d, lens, seed):
    cache = new_cache(n_seq, 1, 2, cap, d)
    st = wl.TokenStream("student_t", cache.units, d, device="cuda", seed=seed)
    wl.fill_rows(st, units_view(cache.k), units_view(cache.v), cap)
    cache.len.copy_(torch.tensor(lens, dtype=torch.int32))
    return cache


def test_block_eviction_at_the_largest_capacity(orc):
    d, cap, N = 64, 65536, 40000
    cache = filled(1, cap, d, [cap], seed=81)
    pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    us = cache.unit_shape()
    kept = torch.empty(us + (N,), dtype=torch.int32, device="cuda")
    scores = torch.empty(us + (cap,), dtype=torch.float32, device="cuda")
    vd.vd_evict_block(cache, N, None, 0, oracle.L2, vd.VD_MU_RECOMPUTE, None, kept, scores)
    assert vd.vd_get_device_status() == 0
    post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    kh, sh = kept.view(cache.units, N).cpu().numpy(), scores.view(cache.units, cap).cpu().numpy()
    assert kh.max() > 32767                              # slot indices above 2^15 round-trip
    for u in range(cache.units):
        check_event(orc, oracle.L2, pre_k[u], pre_v[u], post_k[u], post_v[u], cap, N,
                    kept_gpu=kh[u], scores_gpu=sh[u], new_len=int(cache.len[0]))


def test_block_capacity_beyond_the_slot_lists_is_rejected():
    cache = new_cache(1, 1, 1, 65537, 8)
    cache.len.fill_(65537)
    with pytest.raises(vd.VdError) as e:
        vd.vd_evict_block(cache, 100)
    assert e.value.code == 3                              # VD_ERR_UNSUPPORTED, nothing launched
    assert int(cache.len[0]) == 65537


def test_decode_beyond_the_block_limit(orc):
    d, N = 64, 100000                                     # decode keeps no slot list
    cache = filled(1, N + 1, d, [N + 1], seed=82)
    pre_k, pre_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    us = cache.unit_shape()
    ev = torch.empty(us, dtype=torch.int32, device="cuda")
    kept = torch.empty(us + (N,), dtype=torch.int32, device="cuda")
    vd.vd_evict_decode(cache, N, None, oracle.L2, vd.VD_MU_RECOMPUTE, None, ev, kept)
    assert vd.vd_get_device_status() == 0
    post_k, post_v = bits(units_view(cache.k)), bits(units_view(cache.v))
    kh = kept.view(cache.units, N).cpu().numpy()
    for u in range(cache.units):
        check_event(orc, oracle.L2, pre_k[u], pre_v[u], post_k[u], post_v[u], N + 1, N,
                    kept_gpu=kh[u], new_len=int(cache.len[0]))
        missing = sorted(set(range(N + 1)) - set(kh[u].tolist()))
        assert [int(ev.view(-1)[u])] == missing


def test_empty_sequences():
    d, cap, N = 64, 96, 64
    cache = filled(3, cap, d, [0, 90, 0], seed=83)
    us = cache.unit_shape()
    before_k, before_v = cache.k.clone(), cache.v.clone()
    scores = torch.full(us + (cap,), float("nan"), device="cuda")
    vd.vd_score(cache, vd.VD_SCORE_L2, scores)
    assert vd.vd_get_device_status() == 0
    s = scores.view(3, -1, cap)
    assert torch.all(torch.isnan(s[0])) and torch.all(torch.isnan(s[2]))   # nothing to score
    assert not torch.any(torch.isnan(s[1, :, :90]))
    kept = torch.full(us + (N,), -7, dtype=torch.int32, device="cuda")
    vd.vd_evict_block(cache, N, None, 0, vd.VD_SCORE_L2, vd.VD_MU_RECOMPUTE, None, kept)
    assert vd.vd_get_device_status() == 0
    assert cache.len.cpu().tolist() == [0, N, 0]
    k = kept.view(3, -1, N).cpu()
    assert torch.all(k[0] == -1) and torch.all(k[2] == -1)                 # identity of nothing
    for sidx in (0, 2):                                                    # untouched
        assert torch.equal(cache.k[sidx].view(torch.int16), before_k[sidx].view(torch.int16))
        assert torch.equal(cache.v[sidx].view(torch.int16), before_v[sidx].view(torch.int16))
    # a decode step appends into the empty sequences and evicts in the full one
    st = wl.TokenStream("student_t", cache.units, d, device="cuda", seed=84)
    k1, v1 = st.next(1)
    ev = torch.full(us, -7, dtype=torch.int32, device="cuda")
    vd.vd_append_evict_decode(cache, k1.view(us + (1, d)).contiguous(),
                              v1.view(us + (1, d)).contiguous(), N, None, vd.VD_SCORE_L2,
                              vd.VD_MU_RECOMPUTE, None, ev)
    assert vd.vd_get_device_status() == 0
    assert cache.len.cpu().tolist() == [1, N, 1]
    e = ev.view(3, -1).cpu()
    assert torch.all(e[0] == -1) and torch.all(e[2] == -1) and torch.all(e[1] >= 0)
    assert torch.equal(cache.v[0, :, :, 0].view(torch.int16),
                       v1.view(us + (d,))[0].view(torch.int16))
