"""Free-running trajectories (informational): a whole prompt of block prompt
processing (Sec. 2.2 Eq. block_processing) through the CUDA path, exactly as
the benchmark runs it (fused append and eviction, running mean), and through
the oracle's own loop (recomputed fp64 mean, oracle.block_process order),
without ever copying one side's cache into the other.  For every sampled
unit the surviving token positions are compared after every event.

Step-locked parity (the other GPU tests) is the acceptance test: near ties
that fp32 may order either way can legitimately fork a trajectory, after
which the two caches hold different tokens.  This test reports how long the
trajectories agree (printed in the session summary) and asserts only what
must hold: up to the first divergence both sides saw the same cache, so the
first divergent tokens must lie in the near-tie band of that event's oracle
scores.  Needs a GB300."""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle
import paper_2609_23314_gb300 as vd
from paper_2609_23314_gb300 import build, workloads as wl
from vd_gpu import TRAJECTORIES, bits, near_tie_band, units_view

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build.build()
    vd.load_library()
    torch.cuda.set_device(0)
    yield
    assert vd.vd_get_device_status() == 0


@pytest.mark.parametrize("name,n_sample", [("tiny_prefill", 2), ("prefill_gqa8b", 4)])
def test_free_running_trajectory(orc, name, n_sample):
    _, cfg = wl.config(name)
    d, N, B, T = cfg["head_dim"], cfg["N"], cfg["B"], cfg["T"]
    cache = vd.Cache.empty(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], N + B, d)
    U, us = cache.units, cache.unit_shape()
    rng = np.random.default_rng(7)
    sample = sorted(rng.choice(U, size=min(n_sample, U), replace=False).tolist())
    idx = torch.tensor(sample, device="cuda", dtype=torch.long)
    st = wl.stream_for(cfg)
    rs = torch.zeros(us + (d,), dtype=torch.float64, device="cuda")
    kept = torch.empty(us + (N,), dtype=torch.int32, device="cuda")
    gpu_pos = [np.empty(0, np.int64) for _ in sample]
    ora = [(np.empty((0, d), np.uint16), np.empty((0, d), np.uint16), np.empty(0, np.int64))
           for _ in sample]
    first_div, events, same_events = None, 0, 0
    for i in range(T // B):
        k, v = st.next(B)
        k, v = k.view(us + (B, d)).contiguous(), v.view(us + (B, d)).contiguous()
        kb = bits(k.view(U, B, d)[idx])
        vb = bits(v.view(U, B, d)[idx])
        n_before = int(cache.len[0])
        vd.vd_append_evict_block(cache, k, v, B, N, None, vd.VD_SCORE_L2, vd.VD_MU_RUNNING, rs,
                                 kept_idx_out=kept)
        new_pos = np.arange(i * B, (i + 1) * B)
        evicting = n_before + B > N
        kh = kept.view(U, N)[idx].cpu().numpy() if evicting else None
        events += int(evicting)
        all_same = True
        for j, u in enumerate(sample):
            pos = np.concatenate([gpu_pos[j], new_pos])
            gpu_pos[j] = pos[kh[j]] if evicting else pos
            kc, vc, po = ora[j]
            kc, vc, po = np.concatenate([kc, kb[j]]), np.concatenate([vc, vb[j]]), \
                np.concatenate([po, new_pos])
            s = None
            if vc.shape[0] > N:
                kc2, vc2, ko, s = orc.evict_unit(kc, vc, N, oracle.L2)
                pre_po = po
                kc, vc, po = kc2, vc2, po[ko]
            ora[j] = (kc, vc, po)
            if not np.array_equal(np.sort(gpu_pos[j]), np.sort(po)):
                all_same = False
                if first_div is None:
                    # both sides held the same cache before this event: the
                    # tokens they kept differently are near ties of it
                    first_div = (i, u)
                    diff = np.setxor1d(gpu_pos[j], po)
                    slots = np.flatnonzero(np.isin(pre_po, diff))
                    assert s is not None
                    assert np.all(near_tie_band(s, N)[slots]), (name, i, u, diff[:8])
        same_events += int(all_same and first_div is None and evicting)
    assert vd.vd_get_device_status() == 0
    assert int(cache.len[0]) == N
    final = np.mean([len(np.intersect1d(g, o[2])) / N for g, o in zip(gpu_pos, ora)])
    TRAJECTORIES[name] = {"events": events, "units": len(sample),
                          "identical_events": same_events,
                          "first_divergence": first_div, "final_overlap": final}
    if first_div is None:
        # no divergence: the final caches hold the same tokens, byte for byte
        for j, u in enumerate(sample):
            order = np.argsort(gpu_pos[j])
            kc, vc, po = ora[j]
            oo = np.argsort(po)
            assert np.array_equal(bits(units_view(cache.v)[u, :N])[order], vc[oo])
            assert np.array_equal(bits(units_view(cache.k)[u, :N])[order], kc[oo])
