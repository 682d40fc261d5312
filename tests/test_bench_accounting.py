"""The benchmark's host-side accounting (moved rows, algorithmic bytes, the
ncu traffic lookup) and its CPU reference arm; CPU only."""
from __future__ import annotations

import contextlib
import io
import json
import os
import sys

import numpy as np
import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def ordered_kept(n, N, evicted):
    """Slots kept by an ordered eviction, -1 padded to N."""
    kept = [r for r in range(n) if r not in evicted][:N]
    return kept + [-1] * (N - len(kept))


def holefill_kept(n, N, evicted):
    """Slot map of the hole-fill layout: kept rows at or above N fill the
    evicted slots below N in ascending order; other slots keep their row."""
    if n <= N:
        return list(range(n)) + [-1] * (N - n)
    movers = [r for r in range(N, n) if r not in evicted]
    holes = [r for r in range(N) if r in evicted]
    assert len(movers) == len(holes)
    out = list(range(N))
    for h, m in zip(holes, movers):
        out[h] = m
    return out


def fake(cls, U, N, B, d, holefill, mu=1, attn=False):
    w = object.__new__(cls)
    w.torch, w.device, w.U, w.N, w.B, w.d = torch, torch.device("cpu"), U, N, B, d
    w.holefill, w.mu, w.attn = holefill, mu, (object() if attn else None)
    return w


@pytest.mark.parametrize("holefill", [False, True], ids=["ordered", "holefill"])
def test_prefill_moved_rows(holefill):
    rng = np.random.default_rng(3)
    U, N, B = 6, 40, 9
    w = fake(bench.Prefill, U, N, B, 8, holefill)
    kept_list, want = [], 0
    for _ in range(3):
        rows = []
        for u in range(U):
            n = N + B if u != 5 else N - 7           # one unit below budget: nothing moves
            ev = set(rng.choice(n, size=n - N, replace=False).tolist()) if n > N else set()
            k = holefill_kept(n, N, ev) if holefill else ordered_kept(n, N, ev)
            rows.append(k)
            if n > N:
                want += len([h for h in ev if h < N]) if holefill else max(0, N - min(ev))
        kept_list.append(torch.tensor(rows, dtype=torch.int32))
    assert w.moved_rows(kept_list) == pytest.approx(want / 3)


@pytest.mark.parametrize("holefill", [False, True], ids=["ordered", "holefill"])
def test_decode_moved_rows(holefill):
    U, N = 5, 30
    w = fake(bench.Decode, U, N, 1, 8, holefill)
    e = torch.tensor([0, 7, N, -1, N - 1], dtype=torch.int32)   # N: the new token itself
    want = (1 + 1 + 0 + 0 + 1) if holefill else (N + (N - 7) + 0 + 0 + 1)
    assert w.moved_rows([e, e]) == want


def test_bytes_per_launch():
    U, N, B, d = 4, 100, 20, 64
    w = fake(bench.Prefill, U, N, B, d, False, attn=True)
    alg, nominal = w.bytes_per_launch(37)
    v_read = U * (N + B) * d * 2
    state = U * d * 8 * 2 + U * (N + B) * 4
    assert alg == v_read + 37 * d * 8 + state
    assert nominal == v_read + U * N * d * 8 + state
    wd = fake(bench.Decode, U, N, 1, d, True, mu=0)
    alg, nominal = wd.bytes_per_launch(3)
    assert alg == U * (N + 1) * d * 2 + 3 * d * 8 + U * N * 4 + 3 * 4
    assert nominal == U * (N + 1) * d * 2 + U * d * 8 + U * N * 4 + 3 * 4


def test_traffic_is_reported_only_for_the_captured_sources(monkeypatch):
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        t = json.load(f)
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: t["prefill_wide"]["source_hash"])
    assert bench.ncu_traffic("prefill_wide") == t["prefill_wide"]["dram_bytes_per_launch"]
    assert bench.ncu_traffic("no_such_workload") is None
    e = t["prefill_wide"]
    # the same kernel, units and mean mode as the capture, or nothing
    assert bench.ncu_traffic("prefill_wide", kernel=e["kernel"], units=e["units"],
                             mu=e["mu"]) == e["dram_bytes_per_launch"]
    assert bench.ncu_traffic("prefill_wide", units=e["units"] // 2) is None
    assert bench.ncu_traffic("prefill_wide", kernel=e["kernel"].replace("<0,", "<1,")) is None
    # the recomputed mean has an entry of its own
    r = t["prefill_wide:recompute"]
    assert bench.ncu_traffic("prefill_wide", mu="recompute") == r["dram_bytes_per_launch"]
    assert r["mu"] == "recompute" and r["dram_bytes_per_launch"] != e["dram_bytes_per_launch"]
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: "changed")
    assert bench.ncu_traffic("prefill_wide") is None


def test_reference_arm_runs_on_cpu(monkeypatch):
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.main(["--impl", "reference", "--workload", "tiny_prefill", "--steps", "1",
                    "--warmup", "3"])
    line = json.loads(out.getvalue().strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["steps"] == 1
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["higher_is_better"] is True


class _DoneProc:
    """Stands in for the nvidia-smi child process of a ClockSampler."""

    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def test_clock_sampler_window():
    """Samples count from the start of the timed region to the end of the
    untimed run-on; the idle samples before are left out; the timed region's
    own count is reported; any active slowdown reason is kept."""
    cs = bench.ClockSampler(0)
    cs.proc = _DoneProc()
    row = "{},2070,0x0,Not Active,Not Active,Not Active,{}"
    cs.lines = [(0.5, row.format(1200, "Not Active")),             # idle, before
                (1.00, row.format(2070, "Not Active")),            # timed region
                (1.02, row.format(2070, "Not Active")),
                (1.10, row.format(2040, "Active")),                # run-on
                (1.30, row.format(2070, "Not Active")),
                (2.00, row.format(900, "Not Active"))]             # after
    cs.mark(0.99, 1.03, 1.31)
    out = cs.stop()
    assert out["samples"] == 4
    assert out["samples_in_timed_region"] == 2
    assert out["sm_mhz"] == 2070.0 and out["sm_max_mhz"] == 2070.0
    assert out["reasons"] == ["sw_power_cap"]
    assert "read-only" in out["window"]


def test_clock_sampler_without_samples_in_window():
    """No sample inside the window: the last three are reported instead."""
    cs = bench.ClockSampler(0)
    cs.proc = _DoneProc()
    row = "2070,2070,0x0,Not Active,Not Active,Not Active,Not Active"
    cs.lines = [(5.0, row), (5.1, row), (5.2, row), (5.3, row)]
    cs.mark(1.0, 1.01, 1.02)
    out = cs.stop()
    assert out["samples"] == 3 and out["samples_in_timed_region"] == 0


def test_ratio_budget_accounting():
    """Ratio budget: only the steps over their budget evict and count; rows
    move from the evicted slot up to the step's own budget; the steps that
    only append copy their new K and V rows in."""
    U, d = 3, 8
    w = object.__new__(bench.RatioDecode)
    w.torch, w.U, w.N, w.d, w.mu = torch, U, 12, d, 1
    w.record = [(11, 10), (11, 10), (11, 11), (12, 11)]    # n, N_t: the third step appends only
    e = [torch.tensor(x, dtype=torch.int32) for x in ([0, 4, 10], [9, -1, 2], [-1, -1, -1],
                                                       [11, 0, 5])]
    assert w.moved_rows(e) == pytest.approx(((10 + 6 + 0) + (1 + 0 + 8) + 0 + (0 + 11 + 6)) / 4)
    assert w.head_tokens_per_step() == pytest.approx(U * (11 + 11 + 12) / 4)
    alg, nominal = w.bytes_per_launch(10.0)
    v_read = U * d * 2 * (11 + 11 + 12) / 4
    copy_in = U * d * 2 * 2 * 2 * 1 / 4
    assert alg == pytest.approx(v_read + 10.0 * d * 8 + copy_in + U * d * 16)
    assert nominal == pytest.approx(v_read + U * d * 8 * (10 + 10 + 11) / 4 + copy_in + U * d * 16)
    assert set(w.breakdown) == {"scored_rows_read", "moved_rows_rw", "other"}


def test_stricter_fractions():
    r = bench.stricter({"achieved": 7300.0, "peak": 6789.0, "frac": 7300.0 / 6789.0}, 7100.0)
    assert r["above_copy_peak"] is True
    assert r["frac_of_read_peak"] == pytest.approx(7300 / 7100)
    assert r["frac_strict"] == pytest.approx(7300 / bench.NOMINAL_HBM_GBS)
    r = bench.stricter({"achieved": 5000.0, "peak": 6789.0, "frac": 5000 / 6789}, 8000.0)
    assert r["above_copy_peak"] is False and r["frac_strict"] == pytest.approx(5000 / 8000)


def test_cpu_model_names_arm_parts():
    grace = "processor\t: 0\nBogoMIPS\t: 2000.00\nCPU implementer\t: 0x41\nCPU part\t: 0xd4f\n"
    assert bench.cpu_model(grace).startswith("Arm Neoverse V2")
    assert bench.cpu_model("model name\t: Some x86 CPU @ 2.0GHz\n") == "Some x86 CPU @ 2.0GHz"
    assert bench.cpu_model("CPU implementer\t: 0x51\nCPU part\t: 0x001\n").startswith("part 0x001")


def test_reference_arm_prints_the_workload_config(monkeypatch):
    """Both arms describe the workload with the same config object."""
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        bench.main(["--impl", "reference", "--workload", "tiny_prefill", "--steps", "1",
                    "--warmup", "3"])
    line = json.loads(out.getvalue().strip().splitlines()[-1])
    from paper_2609_23314_gb300 import workloads as wl
    _, cfg = wl.config("tiny_prefill")
    want = bench.workload_config("tiny_prefill", cfg, "running", "l2", "ordered", True, False)
    assert line["config"] == json.loads(json.dumps(want))
    for k in ("n_seq", "n_layer", "n_kv_head", "head_dim", "T", "B", "N"):
        assert line["config"][k] == cfg[k]
