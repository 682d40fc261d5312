"""Builds libvd.so in-tree for GB300 (sm_103a) with nvcc.

Each .cu under csrc/ compiles to its own object in parallel, then nvcc links
them into ``paper_2609_23314_gb300/libvd.so`` (CUDA runtime linked
statically).  Rebuilds only when a source or header is newer than the
library.

Every compile runs with ``-Xptxas -v`` and the build fails if any kernel gets
a local-memory stack frame or spills registers (``check_resources``): the
kernels are sized to fit their register budget, and a frame is only ever
accepted by listing the kernel in ``ALLOWED_FRAMES``, which is empty.
"""
from __future__ import annotations

import glob
import os
import re
import subprocess
from concurrent.futures import ThreadPoolExecutor

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD_DIR = os.path.join(PKG, "_build")
LIB = os.path.join(PKG, "libvd.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-Wall",
              "-I", INCLUDE, "-I", CSRC] + ARCH


def _extra_defines():
    """Extra -D flags for tuning sweeps (environment VD_NVCC_DEFINES, e.g.
    "-DVD_RING_ITEMS=3"); empty by default."""
    return [f for f in os.environ.get("VD_NVCC_DEFINES", "").split() if f.startswith("-D")]


# Kernels (mangled names) allowed a stack frame or spills.  Empty: no kernel
# may use local memory.
ALLOWED_FRAMES: frozenset = frozenset()

_ENTRY = re.compile(r"Compiling entry function '([^']+)'")
_FRAME = re.compile(r"(\d+) bytes stack frame, (\d+) bytes spill stores, (\d+) bytes spill loads")
_REGS = re.compile(r"Used (\d+) registers")


def parse_resources(ptxas_log: str) -> dict:
    """ptxas -v output -> {kernel: (registers, stack frame, spill stores,
    spill loads)} for every entry function compiled."""
    out, cur, frame = {}, None, None
    for line in ptxas_log.splitlines():
        m = _ENTRY.search(line)
        if m:
            cur, frame = m.group(1), None
            continue
        m = _FRAME.search(line)
        if m and cur:
            frame = tuple(int(x) for x in m.groups())
            continue
        m = _REGS.search(line)
        if m and cur and frame is not None:
            out[cur] = (int(m.group(1)),) + frame
            cur, frame = None, None
    return out


def check_resources(resources: dict, allowed=ALLOWED_FRAMES) -> list:
    """Kernels with a stack frame or spills that are not allowed."""
    return sorted(k for k, (_, frame, st, ld) in resources.items()
                  if (frame or st or ld) and k not in allowed)


def _nvcc() -> str:
    cand = os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"), "bin", "nvcc")
    return cand if os.path.exists(cand) else "nvcc"


def sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _inputs():
    return sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h"))


def _stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(p) > t for p in _inputs())


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile (if needed) and return the path of libvd.so."""
    if not force and not _stale():
        return LIB
    os.makedirs(BUILD_DIR, exist_ok=True)
    nvcc = _nvcc()

    def compile_one(src):
        obj = os.path.join(BUILD_DIR, os.path.basename(src)[:-3] + ".o")
        cmd = [nvcc] + NVCC_FLAGS + _extra_defines() + ["-Xptxas", "-v", "-c", src, "-o", obj]
        if verbose:
            print(" ".join(cmd), flush=True)
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}{r.stderr}")
        return obj, parse_resources(r.stdout + r.stderr)

    with ThreadPoolExecutor(max_workers=min(8, os.cpu_count() or 1)) as ex:
        done = list(ex.map(compile_one, sources()))
    objs = [o for o, _ in done]
    resources = {}
    for _, res in done:
        resources.update(res)
    bad = check_resources(resources)
    if bad:
        raise RuntimeError("kernels with a stack frame or register spills: " + ", ".join(
            f"{k} {resources[k]}" for k in bad))
    if verbose:
        for k in sorted(resources):
            print(f"  {k}: {resources[k][0]} registers, no local memory", flush=True)
    tmp = LIB + ".tmp"
    cmd = [nvcc, "-shared", "-o", tmp] + objs + ARCH
    if verbose:
        print(" ".join(cmd), flush=True)
    subprocess.run(cmd, check=True)
    os.replace(tmp, LIB)
    return LIB


if __name__ == "__main__":
    print(build(force=True, verbose=True))
