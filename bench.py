"""Benchmark of the ValueDiff eviction hot path on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl vd|reference]
                    [--workload prefill_wide|decode_batched|prefill_gqa8b|ratio_budget|tiny_prefill]

One step = one eviction event of the whole hot path over every unit of the
workload: the block (or token) append of Eq. (block_processing) followed by
pi_N (mean -> scores -> top-N -> in-place K/V compaction).  The workload is
at steady state (cache at N before each append), inputs are resident in HBM
and larger than L2.  Prints one JSON line (rank 0):

  value       head-tokens scored and compacted per second, whole job
  roofline    the fused eviction kernel: algorithmic bytes per launch / its
              CUDA-event duration, against the measured HBM copy bandwidth
  e2e         the same metric through the C ABI with the step's new K/V rows
              copied from pinned host memory (a pool of E2E_POOL staging
              buffers) and the step's result (kept or evicted slots) copied
              back, every step
  cpu_baseline  the fp64 CPU oracle on a bounded sample of the same events
  secondary   the largest decode workload measured the same way (default run)

--impl reference times the oracle itself (the CPU reference of this build).
Multi-GPU (torchrun): every rank runs its own replica of the workload (units
are independent; no collective on the data path) -> weak scaling; the step
time is the max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "cache tokens scored+compacted/s; HBM GB/s as % of GB300 peak per eviction"
UNIT = "head-tokens/s"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 7900.0   # GB300 HBM3e, nominal (context and the strict fraction)
L2_BYTES = 129 * 2 ** 20
# pinned host staging buffers the e2e run cycles through, as a caller's
# staging pool would: copies from 50 distinct 88 MB pinned blocks (4.4 GB)
# ran 4-6x slower than from 8 on the same GB300, although each copy alone
# runs at ~204 GB/s; the buffers are warmed before the timed region
E2E_POOL = 8
CLOCK_TAIL_S = 0.3   # untimed read-only load after the timed region while clocks are sampled


# ---------------------------------------------------------------------------
# host logic shared by all ranks (tested on CPU with gloo)
# ---------------------------------------------------------------------------
def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return ws, rank, local


def rank_seed(base: int, rank: int) -> int:
    """Each rank's replica draws its own inputs."""
    return base + 1000 * rank


def max_over_ranks(value: float, device=None) -> float:
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return value
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(device=None):
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        if device is not None and str(device).startswith("cuda"):
            dist.barrier(device_ids=[device.index if hasattr(device, "index") else 0])
        else:
            dist.barrier()


def nvml_id(device_index: int) -> str:
    """The GPU's id for `nvidia-smi -i`: its UUID, since CUDA and NVML may
    number the GPUs differently (CUDA_VISIBLE_DEVICES, device order); the
    CUDA index where torch does not report a UUID."""
    try:
        import torch
        u = str(torch.cuda.get_device_properties(device_index).uuid)
        if u:
            return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        pass
    return str(device_index)


def bind_to_gpu_numa(gpu_index: int):
    """Pins this process to the host CPUs local to the GPU (sysfs local_cpulist
    of its PCI device), so pinned host buffers are allocated on the GPU's own
    NUMA node; returns the CPU list or None."""
    try:
        bus = subprocess.run(["nvidia-smi", "-i", nvml_id(gpu_index), "--query-gpu=pci.bus_id",
                              "--format=csv,noheader"], capture_output=True, text=True,
                             timeout=20).stdout.strip()
        dom, rest = bus.split(":", 1)
        dev = f"{int(dom, 16):04x}:{rest}".lower()
        with open(f"/sys/bus/pci/devices/{dev}/local_cpulist") as f:
            spec = f.read().strip()
        cpus = set()
        for part in spec.split(","):
            a, _, b = part.partition("-")
            cpus.update(range(int(a), int(b or a) + 1))
        cpus &= os.sched_getaffinity(0)
        if cpus:
            os.sched_setaffinity(0, cpus)
            return spec
    except Exception:
        pass
    return None


def whole_job_rate(units_per_rank_step: float, steps: int, world: int, max_ms: float) -> float:
    return units_per_rank_step * steps * world / (max_ms / 1e3)


# ---------------------------------------------------------------------------
# measured peaks, clocks, ncu traffic
# ---------------------------------------------------------------------------
def hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured (MEASURED_PEAKS.json hbm_gbs)"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback (no MEASURED_PEAKS.json)"


def kernel_source_hash() -> str:
    """Hash of the CUDA sources' code (comments and white space removed), the
    key of the committed ncu traffic: a capture stays valid until the code
    itself changes."""
    import re
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_23314_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(name.encode() + " ".join(text.split()).encode())
    return h.hexdigest()[:16]


def ncu_traffic(workload: str, layout: str = "ordered", separate: bool = False,
                kernel: str | None = None, units: int | None = None, mu: str | None = None):
    """DRAM bytes per launch of the eviction kernel from the committed ncu
    summary, if it was taken on the current kernel sources and (where given)
    for the same kernel instantiation, number of units and mean mode as this
    run; else None.  separate: a prefill step that appends with vd_append
    first (its eviction then finds the new rows in the cache, partly still
    in L2)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            t = json.load(f)
        key = workload if layout == "ordered" else f"{workload}:{layout}"
        key += (":separate" if separate else "") + (":recompute" if mu == "recompute" else "")
        e = t[key]
        if e.get("source_hash") != kernel_source_hash():
            return None
        for field, want in (("kernel", kernel), ("units", units), ("mu", mu)):
            if want is not None and e.get(field) != want:
                return None
        return float(e["dram_bytes_per_launch"])
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self._t = None
        self.window = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", nvml_id(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self._t = threading.Thread(target=self._read, daemon=True)
            self._t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, t0, t1, t2=None):
        """[t0, t1]: the timed region; [t1, t2]: untimed read-only passes over
        the same cache (clock_tail), so that a timed region shorter than a
        few sampling periods still has samples under load."""
        self.window = (t0, t1, t2 if t2 is not None else t1)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self._t:
            self._t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        lines = self.lines
        timed = None
        if self.window is not None:
            t0, t1, t2 = self.window
            timed = sum(1 for ts, _ in lines if t0 <= ts <= t1 + 0.02)
            inside = [ln for ts, ln in lines if t0 <= ts <= t2 + 0.02]
            lines = inside if inside else [ln for _, ln in lines[-3:]]
        else:
            lines = [ln for _, ln in lines]
        for ln in lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[3:7]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        sm.sort()
        out = {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(mx), "reasons": sorted(reasons),
               "samples": len(sm)}
        if timed is not None:
            out["samples_in_timed_region"] = timed
            out["window"] = "timed region + %.2f s of read-only sigma passes over the same cache" % (
                self.window[2] - self.window[1])
        return out


# ---------------------------------------------------------------------------
# workloads at steady state
# ---------------------------------------------------------------------------
class Prefill:
    """Block boundary at steady state: append B rows, evict N + B -> N."""

    def __init__(self, name, cfg, device, seed, mu, variant, n_blocks=8, layout="ordered",
                 score_keys=False, weighted=False, dispersion=False, separate_append=False):
        """n_blocks distinct appended blocks are pre-generated and reused in
        order; the benchmark asks for as many as the prompt has (T / B), so
        every timed event appends rows the cache has not seen.  layout
        "holefill" uses vd_evict_block_holefill with a token-position array.
        The step is one vd_append_evict_block call (the new block read
        straight from its buffer) in either layout, and one
        vd_append_evict_block_ex call with the scoring options;
        separate_append appends with vd_append first."""
        import torch
        import paper_2609_23314_gb300 as vd
        from paper_2609_23314_gb300 import workloads as wl
        self.vd, self.torch = vd, torch
        self.name, self.cfg, self.device = name, cfg, device
        self.N, self.B, self.d = cfg["N"], cfg["B"], cfg["head_dim"]
        self.cap = self.N + self.B
        self.cache = vd.Cache.empty(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], self.cap,
                                    self.d, device=device)
        self.U = self.cache.units
        st = wl.stream_for(cfg, device=str(device), seed=seed)
        kv = self.cache.k.view(self.U, self.cap, self.d), self.cache.v.view(self.U, self.cap, self.d)
        wl.fill_rows(st, kv[0], kv[1], self.N, chunk_units=64)
        self.cache.len.fill_(self.N)
        us = self.cache.unit_shape()
        self.blocks = []
        for _ in range(n_blocks):
            k, v = st.next(self.B)
            self.blocks.append((k.view(us + (self.B, self.d)).contiguous(),
                                v.view(us + (self.B, self.d)).contiguous()))
        self.mu, self.variant = mu, variant
        self.rs = torch.zeros(us + (self.d,), dtype=torch.float64, device=device)
        if mu == vd.VD_MU_RUNNING:   # the running sum of the scored tensor (K for the key side)
            vd.vd_running_sum_init_ex(self.cache, score_keys, self.rs)
        self.kept = None
        self.i = 0
        self.launches_per_step = 4     # append + len add, evict + len clamp
        self.holefill = layout == "holefill"
        if self.holefill:
            self.pos = torch.arange(self.cap, dtype=torch.int32, device=device).repeat(
                self.U).view(us + (self.cap,)).contiguous()
            steps = torch.arange(1 << 14, dtype=torch.int32, device=device)
            self.pos_new_all = (self.N + self.B * steps).view(-1, 1).repeat(
                1, cfg["n_seq"]).contiguous()
        # scoring options (key-side rule; attention weights in [0, 0.9))
        self.score_keys = score_keys
        self.attn = None
        if weighted:
            g = torch.Generator(device=device)
            g.manual_seed(seed + 7)
            self.attn = torch.rand(us + (self.cap,), generator=g, device=device) * 0.9
        # per-unit sigma (Sec. 3.1) of the pre-eviction rows, from the score pass
        self.sigma = torch.empty(us, device=device) if dispersion else None
        self.fused = not separate_append
        if self.fused:
            self.launches_per_step = 2     # fused append + evict, len update
        self.pending = None                # the block the next fused call appends

    def head_tokens_per_step(self):
        return self.U * (self.N + self.B)

    def new_kept_buffers(self, k):
        t = self.torch
        return [t.empty(self.cache.unit_shape() + (self.N,), dtype=t.int32, device=self.device)
                for _ in range(k)]

    def append_next(self):
        k, v = self.blocks[self.i % len(self.blocks)]
        self.i += 1
        if self.fused:
            self.pending = (k, v)          # appended by the eviction call itself
        else:
            self.vd.vd_append(self.cache, k, v, self.B)

    def evict(self, kept=None, scores=None):
        options = self.score_keys or self.attn is not None or self.sigma is not None
        if self.fused and options:
            k, v = self.pending
            self.vd.vd_append_evict_block_ex(self.cache, k, v, self.B, self.N, None, self.variant,
                                             self.mu, self.rs if self.mu else None,
                                             self.score_keys, self.attn, kept, scores,
                                             self.sigma)
        elif self.fused:
            k, v = self.pending
            hf = {}
            if self.holefill:
                hf = dict(pos=self.pos,
                          pos_first_new=self.pos_new_all[(self.i - 1) % self.pos_new_all.shape[0]])
            self.vd.vd_append_evict_block(self.cache, k, v, self.B, self.N, None, self.variant,
                                          self.mu, self.rs if self.mu else None, kept, scores,
                                          **hf)
        elif self.holefill:
            pn = self.pos_new_all[(self.i - 1) % self.pos_new_all.shape[0]]
            self.vd.vd_evict_block_holefill(self.cache, self.N, self.pos, pn, None, self.B,
                                            self.variant, self.mu, self.rs if self.mu else None,
                                            kept, scores)
        elif options:
            self.vd.vd_evict_block_ex(self.cache, self.N, None, self.B, self.variant, self.mu,
                                      self.rs if self.mu else None, self.score_keys, self.attn,
                                      kept, scores, self.sigma)
        else:
            self.vd.vd_evict_block(self.cache, self.N, None, self.B, self.variant, self.mu,
                                   self.rs if self.mu else None, kept, scores)

    def step(self, kept=None, ev=None):
        self.append_next()
        if ev is not None:
            ev[0].record()
        self.evict(kept)
        if ev is not None:
            ev[1].record()

    def moved_rows(self, kept_list):
        """Rows moved per launch, all units: the slots r < N that received
        another row (kept[r] not r, and not -1).  Ordered layout: N - the first
        evicted slot of every unit that evicted; hole-fill: the refilled slots."""
        t = self.torch
        total = 0
        ar = t.arange(self.N, device=self.device, dtype=t.int32)
        for kp in kept_list:
            kk = kp.view(self.U, self.N)
            total += int(((kk != ar) & (kk >= 0)).sum().item())
        return total / max(1, len(kept_list))

    def bytes_per_launch(self, moved_rows_total):
        """(algorithmic, nominal) bytes per launch: V read once, moved K and V
        rows read and written, running-sum state (and, hole-fill, the moved
        rows' positions)."""
        n, d = self.N + self.B, self.d
        v_read = self.U * n * d * 2          # the scored tensor (V, or K for the key-side rule)
        move = moved_rows_total * d * 2 * 2 * 2
        extra = self.U * d * 8 * 2 if self.mu else 0
        if self.attn is not None:
            extra += self.U * n * 4          # the attention weights
        if self.holefill:
            extra += moved_rows_total * 4 + self.U * self.B * 4
        self.breakdown = {"scored_rows_read": v_read, "moved_rows_rw": move, "other": extra}
        if self.holefill:
            return v_read + move + extra, v_read + self.U * self.B * d * 2 * 2 * 2 + extra
        return v_read + move + extra, v_read + self.U * self.N * d * 2 * 2 * 2 + extra

    # e2e through the C ABI with host buffers (see run_e2e)
    def e2e_setup(self, pool):
        t = self.torch
        us = self.cache.unit_shape()
        self.h_in = [(k.cpu().pin_memory(), v.cpu().pin_memory())
                     for k, v in self.blocks[:max(1, min(pool, len(self.blocks)))]]
        self.d_in = [(t.empty(us + (self.B, self.d), dtype=t.bfloat16, device=self.device),
                      t.empty(us + (self.B, self.d), dtype=t.bfloat16, device=self.device))
                     for _ in range(2)]
        self.d_out = [t.empty(us + (self.N,), dtype=t.int32, device=self.device) for _ in range(2)]
        self.h_out = [t.empty(us + (self.N,), dtype=t.int32).pin_memory() for _ in range(2)]
        return 2 * self.d_in[0][0].numel() * 2, self.d_out[0].numel() * 4

    def e2e_h2d(self, i, b):
        hk, hv = self.h_in[i % len(self.h_in)]
        self.d_in[b][0].copy_(hk, non_blocking=True)
        self.d_in[b][1].copy_(hv, non_blocking=True)

    def e2e_compute(self, b):
        self.i += 1
        if self.fused:
            self.pending = self.d_in[b]
        else:
            self.vd.vd_append(self.cache, self.d_in[b][0], self.d_in[b][1], self.B)

    def e2e_evict(self, b):
        self.evict(self.d_out[b])

    def e2e_d2h(self, b):
        self.h_out[b].copy_(self.d_out[b], non_blocking=True)

    # oracle sample: the pre-eviction bytes of a few units at steady state
    def oracle_sample(self, units):
        t = self.torch
        vd = self.vd
        k, v = self.blocks[0]
        vd.vd_append(self.cache, k, v, self.B)
        idx = t.arange(units, device=self.device) * max(1, self.U // units)
        kk = self.cache.k.view(self.U, self.cap, self.d)[idx]
        vv = self.cache.v.view(self.U, self.cap, self.d)[idx]
        vd.vd_evict_block(self.cache, self.N, None, self.B, self.variant, self.mu,
                          self.rs if self.mu else None, None, None)
        return kk, vv, self.N + self.B, self.N


class Decode:
    """Decode step at steady state: append one token, evict N + 1 -> N."""

    def __init__(self, name, cfg, device, seed, mu, variant, n_tokens=8, layout="ordered",
                 separate_append=False):
        """n_tokens distinct appended tokens are pre-generated and reused in
        order (the benchmark asks for the workload's 1024 decode steps).
        layout "holefill" uses the hole-fill layout.  A step is one
        vd_append_evict_decode call (the token read from its buffer), or with
        separate_append vd_append then vd_evict_decode(_holefill)."""
        import torch
        import paper_2609_23314_gb300 as vd
        from paper_2609_23314_gb300 import workloads as wl
        self.vd, self.torch = vd, torch
        self.name, self.cfg, self.device = name, cfg, device
        self.N, self.d = cfg["N"], cfg["head_dim"]
        self.B = 1
        self.cap = self.N + 1
        self.cache = vd.Cache.empty(cfg["n_seq"], cfg["n_layer"], cfg["n_kv_head"], self.cap,
                                    self.d, device=device)
        self.U = self.cache.units
        st = wl.stream_for(cfg, device=str(device), seed=seed)
        kv = self.cache.k.view(self.U, self.cap, self.d), self.cache.v.view(self.U, self.cap, self.d)
        wl.fill_rows(st, kv[0], kv[1], self.N, chunk_units=256, initial=True)
        self.cache.len.fill_(self.N)
        us = self.cache.unit_shape()
        self.tokens = []
        for _ in range(n_tokens):
            k, v = st.next(1)
            self.tokens.append((k.view(us + (1, self.d)).contiguous(),
                                v.view(us + (1, self.d)).contiguous()))
        self.mu, self.variant = mu, variant
        self.rs = torch.zeros(us + (self.d,), dtype=torch.float64, device=device)
        if mu == vd.VD_MU_RUNNING:
            vd.vd_running_sum_init(self.cache, self.rs)
        self.i = 0
        self.fused = not separate_append
        self.pending = None
        self.launches_per_step = 2 if self.fused else 4
        self.holefill = layout == "holefill"
        if self.holefill:
            self.pos = torch.arange(self.cap, dtype=torch.int32, device=device).repeat(
                self.U).view(us + (self.cap,)).contiguous()
            steps = torch.arange(1 << 14, dtype=torch.int32, device=device)
            self.pos_new_all = (self.N + steps).view(-1, 1).repeat(1, cfg["n_seq"]).contiguous()

    def head_tokens_per_step(self):
        return self.U * (self.N + 1)

    def new_kept_buffers(self, k):
        t = self.torch
        return [t.empty(self.cache.unit_shape(), dtype=t.int32, device=self.device)
                for _ in range(k)]

    def append_next(self, k=None, v=None):
        if k is None:
            k, v = self.tokens[self.i % len(self.tokens)]
        self.i += 1
        if self.fused:
            self.pending = (k, v)          # appended by the eviction call itself
        else:
            self.vd.vd_append(self.cache, k, v, 1)

    def evict(self, evicted=None, kept=None, scores=None):
        if self.fused:
            k, v = self.pending
            hf = {}
            if self.holefill:
                hf = dict(pos=self.pos,
                          pos_first_new=self.pos_new_all[(self.i - 1) % self.pos_new_all.shape[0]])
            self.vd.vd_append_evict_decode(self.cache, k, v, self.N, None, self.variant, self.mu,
                                           self.rs if self.mu else None, evicted, kept, scores,
                                           **hf)
        elif self.holefill:
            pn = self.pos_new_all[(self.i - 1) % self.pos_new_all.shape[0]]
            self.vd.vd_evict_decode_holefill(self.cache, self.N, self.pos, pn, None, self.variant,
                                             self.mu, self.rs if self.mu else None, evicted,
                                             kept, scores)
        else:
            self.vd.vd_evict_decode(self.cache, self.N, None, self.variant, self.mu,
                                    self.rs if self.mu else None, evicted, kept, scores)

    def step(self, kept=None, ev=None):
        self.append_next()
        if ev is not None:
            ev[0].record()
        self.evict(kept)
        if ev is not None:
            ev[1].record()

    def moved_rows(self, evicted_list):
        """Rows moved per launch, all units: ordered layout, N - evicted slot
        per unit; hole-fill layout, one row per unit whose evicted slot lies
        below N."""
        total = 0
        for e in evicted_list:
            e = e.long()
            if self.holefill:
                total += int(((e >= 0) & (e < self.N)).sum().item())
            else:  # slots e .. N-1 shift down by one; -1: nothing evicted
                total += int(self.torch.where(e >= 0, self.N - e, 0).sum().item())
        return total / max(1, len(evicted_list))

    def bytes_per_launch(self, moved_rows_total):
        """(algorithmic, nominal) bytes per launch; hole-fill adds the
        positions read for the tie-break (4 B per cached row) and written for
        moved rows."""
        n, d = self.N + 1, self.d
        v_read = self.U * n * d * 2
        move = moved_rows_total * d * 2 * 2 * 2
        extra = self.U * d * 8 * 2 if self.mu else 0
        if self.holefill:
            extra += self.U * self.N * 4 + moved_rows_total * 4
        self.breakdown = {"scored_rows_read": v_read, "moved_rows_rw": move, "other": extra}
        if self.holefill:
            return v_read + move + extra, v_read + self.U * d * 2 * 2 * 2 + extra
        return v_read + move + extra, v_read + self.U * self.N * d * 2 * 2 * 2 + extra

    def e2e_setup(self, pool):
        t = self.torch
        us = self.cache.unit_shape()
        self.h_in = [(k.cpu().pin_memory(), v.cpu().pin_memory())
                     for k, v in self.tokens[:max(1, min(pool, len(self.tokens)))]]
        self.d_in = [(t.empty(us + (1, self.d), dtype=t.bfloat16, device=self.device),
                      t.empty(us + (1, self.d), dtype=t.bfloat16, device=self.device))
                     for _ in range(2)]
        self.d_out = [t.empty(us, dtype=t.int32, device=self.device) for _ in range(2)]
        self.h_out = [t.empty(us, dtype=t.int32).pin_memory() for _ in range(2)]
        return 2 * self.d_in[0][0].numel() * 2, self.d_out[0].numel() * 4

    def e2e_h2d(self, i, b):
        hk, hv = self.h_in[i % len(self.h_in)]
        self.d_in[b][0].copy_(hk, non_blocking=True)
        self.d_in[b][1].copy_(hv, non_blocking=True)

    def e2e_compute(self, b):
        self.i += 1
        if self.fused:
            self.pending = self.d_in[b]
        else:
            self.vd.vd_append(self.cache, self.d_in[b][0], self.d_in[b][1], 1)

    def e2e_evict(self, b):
        self.evict(self.d_out[b])

    def e2e_d2h(self, b):
        self.h_out[b].copy_(self.d_out[b], non_blocking=True)

    def oracle_sample(self, units):
        t = self.torch
        vd = self.vd
        k, v = self.tokens[0]
        vd.vd_append(self.cache, k, v, 1)
        idx = t.arange(units, device=self.device) * max(1, self.U // units)
        kk = self.cache.k.view(self.U, self.cap, self.d)[idx]
        vv = self.cache.v.view(self.U, self.cap, self.d)[idx]
        vd.vd_evict_decode(self.cache, self.N, None, self.variant, self.mu,
                           self.rs if self.mu else None, None, None, None)
        return kk, vv, self.N + 1, self.N


class RatioDecode(Decode):
    """Ratio-budget generation (the last `n_steps` tokens of the workload's
    generation): every step appends one token and evicts to the budget
    N_t = floor(L_t / 4) of the tokens processed so far, passed per sequence
    through N_dev.  The budget grows by one every fourth token, so three steps
    in four evict one row and the fourth only appends.  Steps past n_steps
    keep the final budget (every step evicts)."""

    def __init__(self, name, cfg, device, seed, mu, variant, n_steps=64, layout="ordered",
                 separate_append=False):
        from paper_2609_23314_gb300 import workloads as wl
        import torch
        total = cfg["prompt"] + cfg["gen_tokens"]
        n_steps = max(4, min(n_steps, cfg["gen_tokens"]))
        self.L0 = total - n_steps + 1                  # tokens processed after the first step
        self.N_start = wl.budget_at(cfg, self.L0 - 1)  # the cache length before it
        cfg = dict(cfg, N=wl.budget_at(cfg, total))    # capacity N + 1 at the final budget
        super().__init__(name, cfg, device, seed, mu, variant, n_tokens=n_steps, layout=layout,
                         separate_append=separate_append)
        self.cache.len.fill_(self.N_start)
        if mu == self.vd.VD_MU_RUNNING:
            self.rs.zero_()
            self.vd.vd_running_sum_init(self.cache, self.rs)
        self.budget = [wl.budget_at(cfg, self.L0 + i) for i in range(n_steps)]
        self.N_dev = torch.tensor(self.budget, dtype=torch.int32, device=device).view(
            -1, 1).repeat(1, cfg["n_seq"]).contiguous()
        self.length = self.N_start     # host copy of every sequence's length
        self.record = []               # (n, N_t) of the steps measure_gpu times
        self.recording = False

    def _budget(self):
        return min(self.i - 1, len(self.budget) - 1)

    def evict(self, evicted=None, kept=None, scores=None):
        j = self._budget()
        Nt = self.budget[j]
        n = self.length + 1
        self.length = min(n, Nt)
        if self.recording:
            self.record.append((n, Nt))
        k, v = self.pending if self.fused else (None, None)
        if self.fused:
            self.vd.vd_append_evict_decode(self.cache, k, v, self.N, self.N_dev[j], self.variant,
                                           self.mu, self.rs if self.mu else None, evicted, kept,
                                           scores)
        else:
            self.vd.vd_evict_decode(self.cache, self.N, self.N_dev[j], self.variant, self.mu,
                                    self.rs if self.mu else None, evicted, kept, scores)

    def head_tokens_per_step(self):
        """Head-tokens scored per timed step: the cached rows of the steps
        that evicted (a step at the budget only appends)."""
        rec = self.record or [(self.N + 1, self.N)]
        return self.U * sum(n for n, Nt in rec if n > Nt) / len(rec)

    def moved_rows(self, evicted_list):
        rec = self.record or []
        total = 0
        for e, (n, Nt) in zip(evicted_list, rec):
            e = e.long()
            total += int(self.torch.where(e >= 0, Nt - e, 0).sum().item())
        return total / max(1, len(evicted_list))

    def bytes_per_launch(self, moved_rows_total):
        """Per launch, averaged over the timed steps: V read once on the steps
        that evict, the moved rows, the running sum, and on the steps that only
        append, the new K and V rows copied in (read and written)."""
        rec = self.record or [(self.N + 1, self.N)]
        d = self.d
        ev = [(n, Nt) for n, Nt in rec if n > Nt]
        v_read = self.U * d * 2 * sum(n for n, _ in ev) / len(rec)
        copy_in = self.U * d * 2 * 2 * 2 * (len(rec) - len(ev)) / len(rec)
        move = moved_rows_total * d * 2 * 2 * 2
        extra = self.U * d * 8 * 2 if self.mu else 0
        nominal = v_read + self.U * d * 2 * 2 * 2 * sum(Nt for _, Nt in ev) / len(rec)
        self.breakdown = {"scored_rows_read": v_read, "moved_rows_rw": move,
                          "other": copy_in + extra}
        return v_read + move + copy_in + extra, nominal + copy_in + extra


def make_workload(name, device, seed, mu, variant, n_seq=None, events=8, layout="ordered",
                  **opts):
    """`events` = warm-up + timed steps: that many distinct blocks / tokens are
    pre-generated, up to the workload's own length (T / B blocks of the
    prompt, or its decode steps); longer runs reuse them in order."""
    from paper_2609_23314_gb300 import workloads as wl
    _, cfg = wl.config(name)
    if n_seq:
        cfg["n_seq"] = n_seq
    if cfg["kind"] == "prefill":
        pool = max(8, min(events, cfg["T"] // cfg["B"]))
        return Prefill(name, cfg, device, seed, mu, variant, n_blocks=pool, layout=layout, **opts)
    if cfg["kind"] == "decode":
        pool = max(8, min(events, cfg["steps"]))
        return Decode(name, cfg, device, seed, mu, variant, n_tokens=pool, layout=layout, **opts)
    # ratio budget: the last `events` steps of the generation, budgets growing
    return RatioDecode(name, cfg, device, seed, mu, variant, n_steps=max(8, events),
                       layout=layout, **opts)


# ---------------------------------------------------------------------------
# measurement
# ---------------------------------------------------------------------------
def run_e2e(w, steps, device):
    """Steps through the C ABI with the step's new rows copied in from pinned
    host memory and its result (kept slots, or evicted slots for decode)
    copied back, every step.  Three streams overlap the copies with the
    eviction: copy-in (staging buffer b = step % 2), compute (append from the
    staging buffer and evict, in one call where the step is fused), copy-out;
    events keep a staging or result
    buffer from being reused before its consumer is done.  Returns the time
    from the first copy-in to the last copy-out (ms)."""
    import torch
    comp = torch.cuda.current_stream()
    h2d, d2h = torch.cuda.Stream(), torch.cuda.Stream()
    ev = lambda: torch.cuda.Event()
    copied, free, done, out = [ev(), ev()], [ev(), ev()], [ev(), ev()], [ev(), ev()]
    for b in range(2):
        free[b].record(comp)
        out[b].record(comp)
    barrier(device)
    torch.cuda.synchronize()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(comp)
    h2d.wait_stream(comp)
    d2h.wait_stream(comp)
    for i in range(steps):
        b = i % 2
        with torch.cuda.stream(h2d):
            h2d.wait_event(free[b])
            w.e2e_h2d(i, b)
            copied[b].record(h2d)
        comp.wait_event(copied[b])
        w.e2e_compute(b)
        comp.wait_event(out[b])
        w.e2e_evict(b)
        free[b].record(comp)               # the staging buffer is read up to here
        done[b].record(comp)
        with torch.cuda.stream(d2h):
            d2h.wait_event(done[b])
            w.e2e_d2h(b)
            out[b].record(d2h)
    comp.wait_stream(d2h)
    comp.wait_stream(h2d)
    stop.record(comp)
    torch.cuda.synchronize()
    return start.elapsed_time(stop)


def h2d_rate(w, nbytes, reps=5):
    """GB/s of one step's host-to-device copies alone (the e2e buffers, no
    eviction running): the link rate the e2e number is measured against."""
    import torch
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    times = []
    for i in range(reps + 1):
        torch.cuda.synchronize()
        a.record()
        w.e2e_h2d(i, 0)
        b.record()
        torch.cuda.synchronize()
        if i:
            times.append(a.elapsed_time(b))
    times.sort()
    return nbytes / (times[len(times) // 2] / 1e3) / 1e9


def clock_tail(w, seconds):
    """Keeps the GPU streaming the workload's cache for `seconds` after the
    timed region, so that a timed region shorter than a few sampling periods
    (20 ms) still has clock samples under load.  The passes are read-only
    (vd_score_ex with only the per-unit sigma as output): the cache, its
    length and the running sum stay as the timed steps left them, for the
    measurements that follow."""
    import torch
    sigma = torch.empty(w.cache.unit_shape(), device=w.cache.k.device)
    t0 = time.time()
    while time.time() - t0 < seconds:
        for _ in range(8):
            w.vd.vd_score_ex(w.cache, w.vd.VD_SCORE_L2, False, None, sigma)
        torch.cuda.synchronize()


def measure_gpu(w, steps, warmup, device, e2e_steps):
    import torch
    for _ in range(warmup):
        w.step()
    torch.cuda.synchronize()
    kept = w.new_kept_buffers(steps)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(device)
    torch.cuda.synchronize()
    clocks = ClockSampler(device.index if device.index is not None else 0)
    clocks.start()
    time.sleep(0.5)
    t_begin = time.time()
    w.recording = True
    start.record()
    for i in range(steps):
        w.step(kept[i], evs[i])
    stop.record()
    w.recording = False
    torch.cuda.synchronize()
    t_end = time.time()
    clock_tail(w, CLOCK_TAIL_S)
    clocks.mark(t_begin, t_end, time.time())
    clk = clocks.stop()
    barrier(device)
    step_ms = start.elapsed_time(stop)
    kern_ms = sum(a.elapsed_time(b) for a, b in evs) / steps
    moved = w.moved_rows(kept)
    # end to end through the C ABI with host buffers
    bi, bo = w.e2e_setup(min(e2e_steps, E2E_POOL))
    # a staging pool is long-lived: copy from every buffer twice before timing
    # (a freshly pinned buffer's first copies measured up to 12x slower)
    for i in range(2 * len(w.h_in)):
        w.e2e_h2d(i, i % 2)
    torch.cuda.synchronize()
    link_gbs = h2d_rate(w, bi)
    run_e2e(w, min(3, warmup), device)
    e2e_ms = run_e2e(w, e2e_steps, device)
    status = w.vd.vd_get_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status}: {w.vd.vd_status_string(status)}")
    return dict(step_ms=step_ms, kern_ms=kern_ms, moved=moved, clocks=clk, e2e_ms=e2e_ms,
                bi=bi, bo=bo, link_gbs=link_gbs)


def eager_call_us(w, steps):
    """Host-bound time of one eager step (append + evict through the binding
    and the C ABI) in a plain loop, without the per-step CUDA events that
    measure_gpu records around each launch: what an eager caller pays."""
    import torch
    for _ in range(3):
        w.step()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        w.step()
    torch.cuda.synchronize()
    status = w.vd.vd_get_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status}: {w.vd.vd_status_string(status)}")
    return (time.perf_counter() - t0) / steps * 1e6


def graph_step_us(w, steps, device):
    """Device time of one step (append + evict) with the host out of the
    loop: `steps` steps captured once in a CUDA graph and replayed.  Small
    workloads are otherwise bound by the host's launch rate."""
    import torch
    side = torch.cuda.Stream(device=device)
    side.wait_stream(torch.cuda.current_stream(device))
    with torch.cuda.stream(side):
        for _ in range(3):
            w.step()
    torch.cuda.current_stream(device).wait_stream(side)
    torch.cuda.synchronize(device)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for _ in range(steps):
            w.step()
    for _ in range(3):
        g.replay()
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 20
    torch.cuda.synchronize(device)
    start.record()
    for _ in range(reps):
        g.replay()
    stop.record()
    torch.cuda.synchronize(device)
    status = w.vd.vd_get_device_status()
    if status != 0:
        raise RuntimeError(f"device status {status}: {w.vd.vd_status_string(status)}")
    return start.elapsed_time(stop) * 1e3 / (reps * steps)


def measure_dispersion(args, device, variant, peak, rank):
    """vd_score_ex returning sigma_V per unit (Sec. 3.1) over the workload's
    cache at steady state: one score-only launch per step, the mean taken from
    the running sum the eviction calls keep (the V rows read once: the
    algorithmic bytes); the pass with the mean recomputed (V read twice) is
    timed beside it."""
    import torch
    import paper_2609_23314_gb300 as vd
    from paper_2609_23314_gb300 import workloads as wl
    _, cfg = wl.config(args.workload)
    w = make_workload(args.workload, device, rank_seed(wl.BASE_SEED + cfg["index"], rank),
                      vd.VD_MU_RUNNING, vd.VD_SCORE_L2, args.n_seq, events=8)
    sigma = torch.empty(w.cache.unit_shape(), device=device)
    steps = args.extension_steps

    def timed(mu):
        rs = w.rs if mu == vd.VD_MU_RUNNING else None
        for _ in range(args.warmup):
            vd.vd_score_ex(w.cache, vd.VD_SCORE_L2, False, None, sigma, mu=mu, running_sum=rs)
        start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        start.record()
        for _ in range(steps):
            vd.vd_score_ex(w.cache, vd.VD_SCORE_L2, False, None, sigma, mu=mu, running_sum=rs)
        stop.record()
        torch.cuda.synchronize()
        return max_over_ranks(start.elapsed_time(stop), device) / steps

    ms_re = timed(vd.VD_MU_RECOMPUTE)
    ms = timed(vd.VD_MU_RUNNING)
    kernel = "vd::evict_kernel<0, true, false, false, true> (score only)"
    # the realized sigma_V / sigma_K of the generator (untimed)
    sigma_k = torch.empty_like(sigma)
    vd.vd_score_ex(w.cache, vd.VD_SCORE_L2, True, None, sigma_k)
    ratio = float((sigma / sigma_k).mean().item())
    n = int(w.cache.len[0])
    alg = w.U * n * w.d * 2 + w.U * 4
    achieved = alg / (ms / 1e3) / 1e9
    tr = ncu_traffic("prefill_wide:sigma", kernel=kernel, units=w.U, mu="running")
    tr_re = ncu_traffic("prefill_wide:sigma", kernel=kernel, units=w.U, mu="recompute")
    res = {"value": w.U * n / (ms / 1e3), "step_ms": ms, "mean": "running sum",
           "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                        "frac": achieved / peak, "kernel": kernel, "traffic": tr,
                        "algorithmic_bytes_per_launch": alg, "kernel_ms": ms,
                        "sigma_v_mean": float(sigma.mean().item()),
                        "sigma_k_mean": float(sigma_k.mean().item()),
                        "sigma_v_over_sigma_k": ratio},
           "recomputed_mean": {"value": w.U * n / (ms_re / 1e3), "step_ms": ms_re,
                               "frac_of_peak": alg / (ms_re / 1e3) / 1e9 / peak,
                               "traffic": tr_re,
                               "note": "V read twice (sum, then scores); frac counts it once"}}
    del w
    torch.cuda.empty_cache()
    return res


def cpu_baseline(w, budget_s=2.0, max_units=64):
    """The fp64 oracle (as it stands) on a bounded sample of the same events,
    on every host core; returns the extrapolated head-tokens/s."""
    import numpy as np
    import oracle
    orc = oracle.load()
    cores = os.cpu_count() or 1
    units = min(max_units, w.U)
    kk, vv, n, N = w.oracle_sample(units)
    k0 = kk.contiguous().view(w.torch.int16).cpu().numpy().view(np.uint16).copy()
    v0 = vv.contiguous().view(w.torch.int16).cpu().numpy().view(np.uint16).copy()
    lens = np.full(units, n, np.int32)
    Ns = np.full(units, N, np.int32)
    var = int(w.variant)
    elapsed, events = 0.0, 0
    while elapsed < budget_s or events == 0:
        k, v = k0.copy(), v0.copy()
        t0 = time.perf_counter()
        orc.evict_units(k, v, lens, Ns, 1, var, nthreads=cores)
        elapsed += time.perf_counter() - t0
        events += 1
    rate = units * n * events / elapsed
    # one thread on a smaller sample of the same units
    u1 = min(units, 4)
    k, v = k0[:u1].copy(), v0[:u1].copy()
    t0 = time.perf_counter()
    orc.evict_units(k, v, lens[:u1], Ns[:u1], 1, var, nthreads=1)
    rate1 = u1 * n / (time.perf_counter() - t0)
    return {"value": rate, "unit": UNIT, "cores": cores, "kind": "oracle",
            "single_thread_value": rate1, "cpu_model": cpu_model(),
            "sample": f"{units} of {w.U} units x {events} events of {w.name} at n={n} -> N={N}; "
                      f"fp64 C oracle, one POSIX thread per core, {elapsed:.2f} s wall; "
                      f"single thread: {u1} units x 1 event"}


# Arm Ltd. (implementer 0x41) part numbers of server cores, for hosts whose
# /proc/cpuinfo names no model (Grace reports part 0xd4f)
ARM_PARTS = {"0xd0c": "Arm Neoverse N1", "0xd40": "Arm Neoverse V1", "0xd49": "Arm Neoverse N2",
             "0xd4f": "Arm Neoverse V2", "0xd8e": "Arm Neoverse N3", "0xd84": "Arm Neoverse V3"}


def cpu_model(cpuinfo: str | None = None):
    """The host CPU's model name: x86 'model name', else the Arm core named
    from its implementer and part number in /proc/cpuinfo."""
    if cpuinfo is None:
        try:
            with open("/proc/cpuinfo") as f:
                cpuinfo = f.read()
        except OSError:
            return "unknown"
    fields = {}
    for line in cpuinfo.splitlines():
        if ":" in line:
            k, v = line.split(":", 1)
            fields.setdefault(k.strip(), v.strip())
    for key in ("model name", "Model"):
        if fields.get(key):
            return fields[key]
    part, impl = fields.get("CPU part", "").lower(), fields.get("CPU implementer", "").lower()
    if impl == "0x41" and part in ARM_PARTS:
        return f"{ARM_PARTS[part]} (part {part})"
    return f"part {part}, implementer {impl}" if part else "unknown"


def read_peak(device, gib=4, reps=6):
    """A read-only streaming rate measured in this run (GB/s): the faster of
    torch's int64 and fp32 sums over a buffer larger than L2, best of `reps`
    (on a GB300 these read at ~6.4-6.7 TB/s, a little below the kernels that
    only read, which is why the nominal rate bounds frac_strict).  The copy peak of
    MEASURED_PEAKS.json counts a read and a write per byte moved; kernels
    that mostly read (the score passes, decode) can exceed it, so every
    fraction is also reported against the larger of this and the nominal
    HBM3e rate."""
    import torch
    x = torch.ones(gib * 2 ** 30 // 4, dtype=torch.float32, device=device)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    best = float("inf")
    for i in range(2 * reps):
        torch.cuda.synchronize()
        a.record()
        if i % 2:
            x.sum()
        else:
            x.view(torch.int64).sum()
        b.record()
        torch.cuda.synchronize()
        best = min(best, a.elapsed_time(b))
    del x
    torch.cuda.empty_cache()
    return gib * 2 ** 30 / (best / 1e3) / 1e9


def stricter(roofline, read_gbs):
    """Adds the fractions against the same-run read-only peak and the nominal
    HBM3e rate, the strictest of the three, and a flag when the copy-peak
    fraction exceeds 1 (the kernel reads more than it writes, or finds part of
    its input in L2)."""
    a = roofline["achieved"]
    roofline["frac_of_read_peak"] = a / read_gbs if read_gbs else None
    roofline["frac_of_nominal"] = a / NOMINAL_HBM_GBS
    roofline["frac_strict"] = a / max(roofline["peak"], read_gbs or 0.0, NOMINAL_HBM_GBS)
    roofline["above_copy_peak"] = roofline["frac"] > 1.0
    return roofline


def workload_config(name, cfg, mu_name, variant, layout, fused, decode):
    """The `config` object of a measurement (both arms print the same one)."""
    from paper_2609_23314_gb300 import workloads as wl
    cap = (cfg["N"] + cfg["B"]) if cfg["kind"] == "prefill" else None
    if cfg["kind"] == "decode":
        cap = cfg["N"] + 1
    if cfg["kind"] == "ratio":
        cap = wl.budget_at(cfg, cfg["prompt"] + cfg["gen_tokens"]) + 1
    cache_gib = wl.units_of(cfg) * cap * cfg["head_dim"] * 4 / 2 ** 30
    return {"workload": name, **{k: cfg[k] for k in cfg if k not in ("index", "kind")},
            "mu": mu_name, "variant": variant, "layout": layout,
            "append": (("fused into the eviction (vd_append_evict_decode)" if decode else
                        "fused into the eviction (vd_append_evict_block)")
                       if fused else "vd_append, then the eviction"),
            "l2": f"inputs larger than L2: cache {cache_gib:.2f} GiB of K+V, touched every step",
            "storage": "bf16"}


def run_vd(args):
    import torch
    import paper_2609_23314_gb300 as vd
    from paper_2609_23314_gb300 import build as vd_build
    ws, rank, local = dist_env()
    if ws > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    device = torch.device("cuda", torch.cuda.current_device())
    host_cpus = bind_to_gpu_numa(device.index)
    if rank == 0:
        vd_build.build()
    barrier(device)
    vd.load_library()
    mu = vd.VD_MU_RUNNING if args.mu == "running" else vd.VD_MU_RECOMPUTE
    variant = vd.VARIANTS[args.variant]
    peak, peak_src = hbm_peak()
    read_gbs = max_over_ranks(-read_peak(device), device) * -1.0   # the lowest over ranks
    from paper_2609_23314_gb300 import workloads as wl

    def one(name, steps, layout="ordered", mu_mode=None, **opts):
        _, cfg = wl.config(name)
        if args.n_seq:
            cfg["n_seq"] = args.n_seq
        if args.separate_append:
            opts = dict(opts, separate_append=True)
        mm = mu if mu_mode is None else mu_mode
        e2e_steps = min(steps, args.e2e_steps)
        w = make_workload(name, device, rank_seed(wl.BASE_SEED + cfg["index"], rank), mm,
                          variant, args.n_seq, events=args.warmup + steps + e2e_steps + 4,
                          layout=layout, **opts)
        m = measure_gpu(w, steps, args.warmup, device, e2e_steps)
        step_ms = max_over_ranks(m["step_ms"], device) / steps
        kern_ms = max_over_ranks(m["kern_ms"], device)
        e2e_ms = max_over_ranks(m["e2e_ms"], device) / e2e_steps
        tok = w.head_tokens_per_step()
        alg, nominal = w.bytes_per_launch(m["moved"])
        achieved = alg / (kern_ms / 1e3) / 1e9
        kernel = (f"vd::evict_kernel<{variant}, {str(isinstance(w, Decode)).lower()}, "
                  f"{str(layout == 'holefill').lower()}, "
                  f"{str(getattr(w, 'fused', False)).lower()}>")
        mu_name = "running" if mm == vd.VD_MU_RUNNING else "recompute"
        traffic = None
        if not (set(opts) - {"separate_append"}):   # scoring options: never captured
            traffic = ncu_traffic(name, layout, separate=not getattr(w, "fused", True),
                                  kernel=kernel, units=w.U, mu=mu_name)
        res = {
            "workload": name, "w": w, "m": m, "step_ms": step_ms, "kern_ms": kern_ms,
            "value": tok * ws / (step_ms / 1e3),
            "e2e": {"value": tok * ws / (e2e_ms / 1e3), "unit": UNIT,
                    "h2d_bytes_per_step": m["bi"], "d2h_bytes_per_step": m["bo"],
                    "h2d_gbs_alone": m["link_gbs"]},
            "roofline": stricter({
                "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic, "kernel": kernel,
                "algorithmic_bytes_per_launch": alg, "nominal_bytes_per_launch": nominal,
                "bytes_breakdown": dict(w.breakdown), "moved_rows_per_launch": m["moved"],
                "kernel_ms": kern_ms,
                "peak_source": peak_src + ", of measured" if "measured" in peak_src else peak_src},
                read_gbs),
            "config": workload_config(name, cfg, mu_name, args.variant, layout,
                                      getattr(w, "fused", False), isinstance(w, Decode)),
        }
        if isinstance(w, RatioDecode):
            res["config"]["budgets"] = (f"N_t = floor(L_t / 4), {w.budget[0]}..{w.budget[-1]} "
                                        "over the timed window; 3 of 4 steps evict")
        return res

    def brief(r):
        """The parts of a measurement that go into the JSON line."""
        out = {k: r[k] for k in ("value", "step_ms", "roofline", "e2e")}
        out["mu"] = r["config"]["mu"]
        return out

    def release(r):
        if r is not None:
            r.pop("w", None)
            torch.cuda.empty_cache()

    summary = {}

    def summarize(label, r):
        rf = r["roofline"]
        tr = rf.get("traffic")
        summary[label] = [round(r["kern_ms"], 4), round(rf["frac"], 3), round(rf["frac_strict"], 3),
                          round(tr / rf["algorithmic_bytes_per_launch"], 3) if tr else None,
                          round(r["e2e"]["value"] / 1e9, 3)]

    if args.dispersion_only:
        # the sigma pass alone (score-only launches, both mean modes): a short
        # run whose launches come in a fixed order, for profiling
        disp = measure_dispersion(args, device, variant, peak, rank)
        if rank == 0:
            print(json.dumps({"metric": METRIC, "unit": UNIT, "dispersion": disp}), flush=True)
        return
    primary = one(args.workload, args.steps, args.layout)
    summarize(f"{args.workload} ({primary['config']['mu']} mean)", primary)
    base = None
    if rank == 0 and not args.no_cpu_baseline:
        base = cpu_baseline(primary["w"])
    launches = primary["w"].launches_per_step * args.steps
    release(primary)
    secondary = None
    if args.secondary not in ("", "none") and args.secondary != args.workload:
        secondary = one(args.secondary, args.secondary_steps, args.layout)
        summarize(f"{args.secondary} ({secondary['config']['mu']} mean)", secondary)
        release(secondary)
    # the other configurations (and the paper's recomputed mean, Sec. 3.2
    # Eq. vd, beside the running sum) measured the same way
    configs = {}
    if args.config_steps > 0 and args.layout == "ordered":
        plan = [(n, None) for n in ("prefill_gqa8b", "ratio_budget")
                if n not in (args.workload, args.secondary)]
        other_mu = vd.VD_MU_RECOMPUTE if mu == vd.VD_MU_RUNNING else vd.VD_MU_RUNNING
        plan += [(n, other_mu) for n in (args.workload, "prefill_gqa8b")]
        for name, mm in plan:
            r = one(name, args.config_steps, "ordered", mm)
            label = f"{name} ({r['config']['mu']} mean)"
            configs[label] = brief(r)
            summarize(label, r)
            release(r)
    # the same prefill step with a separate vd_append launch before the
    # eviction (the two-call form), for comparison with the fused step
    separate = None
    if (args.extension_steps > 0 and not args.separate_append and args.layout == "ordered"
            and wl.config(args.workload)[1]["kind"] == "prefill"):
        r = one(args.workload, args.extension_steps, "ordered", separate_append=True)
        separate = {"value": r["value"], "step_ms": r["step_ms"], "kernel_ms": r["kern_ms"],
                    "roofline_frac": r["roofline"]["frac"], "e2e": r["e2e"]["value"]}
        release(r)
    # the smallest workload's per-event latency (a few units: launch- and
    # latency-bound, reported in microseconds)
    latency = None
    if args.latency_steps > 0:
        r = one("tiny_prefill", args.latency_steps)
        latency = {"workload": "tiny_prefill",
                   "event_us": r["step_ms"] * 1e3,
                   "event_us_note": "timed loop with two CUDA events recorded per step",
                   "eager_call_us": eager_call_us(r["w"], 200),
                   "kernel_us": r["kern_ms"] * 1e3, "e2e_event_us":
                   r["w"].head_tokens_per_step() * ws / r["e2e"]["value"] * 1e6,
                   "graph_event_us": graph_step_us(r["w"], args.latency_steps, device)}
        summary["tiny_prefill us/event (eager call, graph)"] = [
            round(latency["eager_call_us"], 2), round(latency["graph_event_us"], 2)]
        release(r)
    # the hole-fill cache layout (a next row: same policy, fewest rows moved)
    holefill = {}
    if args.holefill_steps > 0 and args.layout == "ordered":
        for name in (args.workload, args.secondary, "prefill_gqa8b"):
            if name in ("", "none") or name in holefill:
                continue
            r = one(name, args.holefill_steps, "holefill")
            holefill[name] = brief(r)
            summarize(f"{name} hole-fill", r)
            release(r)
    # scoring options on the primary (prefill) workload: the K-side rule (with
    # the running mean of K, as the primary's of V), attention weights, and the
    # per-unit dispersion sigma_V from a score-only pass, and as a by-product
    # of the eviction's own score pass
    extensions = {}
    if args.extension_steps > 0 and wl.config(args.workload)[1]["kind"] == "prefill":
        for key, opts, mu_mode in (("key_side", dict(score_keys=True), None),
                                   ("attention_weighted", dict(weighted=True), None),
                                   ("dispersion_by_product", dict(dispersion=True), None)):
            r = one(args.workload, args.extension_steps, "ordered", mu_mode, **opts)
            extensions[key] = {"value": r["value"], "step_ms": r["step_ms"],
                               "roofline": r["roofline"]}
            if r["w"].sigma is not None:
                extensions[key]["sigma_v_mean"] = float(r["w"].sigma.mean().item())
            summarize(f"{args.workload} {key}", r)
            release(r)
        disp = measure_dispersion(args, device, variant, peak, rank)
        stricter(disp["roofline"], read_gbs)
        extensions["dispersion"] = disp
        alg_d = disp["roofline"]["algorithmic_bytes_per_launch"]
        tr_d, tr_r = disp["roofline"]["traffic"], disp["recomputed_mean"]["traffic"]
        summary["sigma pass (running, recomputed mean)"] = [
            round(disp["step_ms"], 4), round(disp["roofline"]["frac"], 3),
            round(tr_d / alg_d, 3) if tr_d else None,
            round(disp["recomputed_mean"]["step_ms"], 4),
            round(disp["recomputed_mean"]["frac_of_peak"], 3),
            round(tr_r / alg_d, 3) if tr_r else None]
    if rank == 0:
        line = {
            "metric": METRIC, "value": primary["value"], "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": primary["step_ms"],
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f32", "data": "synthetic (seeded generators shaped like the paper's workloads)",
            "config": primary["config"],
            "roofline": primary["roofline"],
            "e2e": primary["e2e"],
            "clocks": primary["m"]["clocks"],
            "gpu_launches": launches,
            "host_cpus": host_cpus,
            "peaks_gbs": {"copy_measured": peak, "read_only_this_run": read_gbs,
                          "nominal_hbm3e": NOMINAL_HBM_GBS},
        }
        if base is not None:
            line["cpu_baseline"] = base
        if secondary is not None:
            line["secondary"] = {k: secondary[k] for k in ("workload", "value", "step_ms", "roofline",
                                                           "e2e", "config")}
            line["secondary"]["clocks"] = secondary["m"]["clocks"]
        if configs:
            line["configs"] = configs
        if separate is not None:
            line["separate_append"] = separate
        if latency is not None:
            line["latency"] = latency
        if holefill:
            line["holefill_layout"] = holefill
        if extensions:
            line["extensions"] = extensions
        # last, so that a reader of the line's tail sees every configuration
        line["summary"] = {"columns": ["kernel_ms", "frac_of_copy_peak", "frac_strict",
                                       "ncu_traffic_over_algorithmic", "e2e_G_head_tokens_per_s"],
                           **summary}
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_reference(args):
    """The CPU oracle as the reference arm: each step = one oracle pass over a
    bounded sample of the workload's units at steady state."""
    ws, rank, _ = dist_env()
    if rank != 0:
        return
    import numpy as np
    import torch
    import oracle
    from paper_2609_23314_gb300 import workloads as wl
    orc = oracle.load()
    name, cfg = wl.config(args.workload)
    cores = os.cpu_count() or 1
    d = cfg["head_dim"]
    if cfg["kind"] == "prefill":
        N, n = cfg["N"], cfg["N"] + cfg["B"]
    else:
        if cfg["kind"] == "ratio":
            cfg["N"] = wl.budget_at(cfg, cfg["prompt"] + cfg["gen_tokens"])
        N, n = cfg["N"], cfg["N"] + 1
    units = max(1, min(wl.units_of(cfg), cores * 2))
    st = wl.stream_for(cfg, device="cpu", units=units)
    k, v = st.next(n, initial=True)
    k0 = k.view(torch.int16).numpy().view(np.uint16).copy()
    v0 = v.view(torch.int16).numpy().view(np.uint16).copy()
    lens = np.full(units, n, np.int32)
    Ns = np.full(units, N, np.int32)
    var = {"l2": 0, "dir": 1, "norm": 2}[args.variant]
    for _ in range(args.warmup):
        kk, vv = k0.copy(), v0.copy()
        orc.evict_units(kk, vv, lens, Ns, 1, var, nthreads=cores)
    total = 0.0
    for _ in range(args.steps):
        kk, vv = k0.copy(), v0.copy()
        t0 = time.perf_counter()
        orc.evict_units(kk, vv, lens, Ns, 1, var, nthreads=cores)
        total += time.perf_counter() - t0
    ms = total / args.steps * 1e3
    value = units * n / (ms / 1e3)
    _, cfg0 = wl.config(args.workload)
    if args.n_seq:
        cfg0["n_seq"] = args.n_seq
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": workload_config(name, cfg0, args.mu, args.variant, args.layout,
                                      not args.separate_append, cfg0["kind"] != "prefill"),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "cpu_model": cpu_model(),
                             "sample": f"{units} of {wl.units_of(cfg0)} units of {name} per step "
                                       f"at n={n} -> N={N} (fp64 C oracle, one thread per core)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["vd", "reference"], default="vd")
    ap.add_argument("--workload", default="prefill_wide")
    ap.add_argument("--secondary", default="decode_batched",
                    help="a second workload measured into the same line ('' to skip)")
    ap.add_argument("--secondary-steps", type=int, default=50)
    ap.add_argument("--layout", choices=["ordered", "holefill"], default="ordered",
                    help="cache layout of the primary and secondary measurements")
    ap.add_argument("--extension-steps", type=int, default=50,
                    help="steps of the key-side / weighted / dispersion measurements (0: skip)")
    ap.add_argument("--holefill-steps", type=int, default=50,
                    help="steps of the extra hole-fill-layout measurements (0: skip)")
    ap.add_argument("--config-steps", type=int, default=50,
                    help="steps of the other configurations and the other mean mode (0: skip)")
    ap.add_argument("--separate-append", action="store_true",
                    help="prefill steps append with vd_append, then evict (default: one "
                         "vd_append_evict_block call)")
    ap.add_argument("--mu", choices=["running", "recompute"], default="running")
    ap.add_argument("--variant", choices=["l2", "dir", "norm"], default="l2")
    ap.add_argument("--e2e-steps", type=int, default=50)
    ap.add_argument("--latency-steps", type=int, default=12,
                    help="events of the tiny_prefill latency measurement (0: skip)")
    ap.add_argument("--n-seq", type=int, default=None,
                    help="override the workload's number of sequences (smaller profiling cases)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--dispersion-only", action="store_true",
                    help="time only the sigma pass of the workload (profiling runs)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    if args.steps is None:
        # prefill_wide: 200 evicting block events of its 240 (all distinct blocks)
        args.steps = 5 if args.impl == "reference" else 200
    if args.impl == "reference":
        run_reference(args)
    else:
        run_vd(args)


if __name__ == "__main__":
    main()
