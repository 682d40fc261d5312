"""fp64 CPU oracle for ValueDiff KV-cache eviction -- TEST INFRASTRUCTURE ONLY.

The plain, slow, obviously-correct reference that the CUDA library is checked
against.  Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU
baseline may import it; the library itself never does, and this package never
imports the library.  The arithmetic lives in ``vd_oracle.c`` (fp64, plain
loops); this module only marshals numpy arrays and drives events in the order
the paper states them:

* ``scores`` / ``mean`` / ``select_top_n`` / ``evict_unit`` -- Sec. 3.2
  Eq. (vd) and Sec. 2.1 Eq. (eviction).
* ``block_process`` -- Sec. 2.2 Eq. (block_processing): append a block of B
  tokens, then apply pi_N; B = T is standard eviction, B = 1 is per-token.

Inputs are bf16 bit patterns as ``numpy.uint16`` arrays shaped [n, d].
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

L2, DIR, NORM = 0, 1, 2
VARIANTS = {"l2": L2, "dir": DIR, "norm": NORM}

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "vd_oracle.c")
_HDR = os.path.join(_HERE, "vd_oracle.h")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile the oracle with gcc (-O2, no fast-math: IEEE fp64 throughout)."""
    stale = (not os.path.exists(out)) or any(
        os.path.getmtime(p) > os.path.getmtime(out) for p in (src, _HDR))
    if force or stale:
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
               "-ffp-contract=off", "-I", _HERE, src, "-o", out, "-lm", "-lpthread"]
        subprocess.run(cmd, check=True)
    return out


def _bind(lib: ctypes.CDLL) -> ctypes.CDLL:
    p = ctypes.c_void_p
    i64 = ctypes.c_int64
    lib.vdo_bf16_to_double.argtypes = [ctypes.c_uint16]
    lib.vdo_bf16_to_double.restype = ctypes.c_double
    lib.vdo_sum_rows.argtypes = [p, i64, i64, p]
    lib.vdo_sum_rows.restype = None
    lib.vdo_mean.argtypes = [p, i64, i64, p]
    lib.vdo_mean.restype = None
    lib.vdo_scores.argtypes = [p, i64, i64, ctypes.c_int, p]
    lib.vdo_scores.restype = None
    lib.vdo_scores_weighted.argtypes = [p, i64, i64, ctypes.c_int, p, p]
    lib.vdo_scores_weighted.restype = None
    lib.vdo_dispersion.argtypes = [p, i64, i64]
    lib.vdo_dispersion.restype = ctypes.c_double
    lib.vdo_select_top_n.argtypes = [p, i64, i64, p]
    lib.vdo_select_top_n.restype = i64
    lib.vdo_evict_unit.argtypes = [p, p, i64, i64, i64, ctypes.c_int, p, p]
    lib.vdo_evict_unit.restype = i64
    lib.vdo_evict_units.argtypes = [p, p, p, p, i64, i64, i64, i64, ctypes.c_int, p, i64,
                                    ctypes.c_int]
    lib.vdo_evict_units.restype = ctypes.c_int
    return lib


class Oracle:
    """Thin numpy front end over one compiled copy of the oracle."""

    def __init__(self, path: str):
        self.path = path
        self.lib = _bind(ctypes.CDLL(path))

    # -- helpers ----------------------------------------------------------
    @staticmethod
    def _u16(a) -> np.ndarray:
        a = np.ascontiguousarray(a)
        if a.dtype != np.uint16:
            raise TypeError("oracle inputs are bf16 bit patterns (numpy.uint16)")
        return a

    @staticmethod
    def _ptr(a: np.ndarray):
        return a.ctypes.data_as(ctypes.c_void_p)

    # -- Eq. (vd) ---------------------------------------------------------
    def sum_rows(self, v) -> np.ndarray:
        v = self._u16(v)
        n, d = v.shape
        out = np.empty(d, np.float64)
        self.lib.vdo_sum_rows(self._ptr(v), n, d, self._ptr(out))
        return out

    def mean(self, v) -> np.ndarray:
        v = self._u16(v)
        n, d = v.shape
        out = np.empty(d, np.float64)
        self.lib.vdo_mean(self._ptr(v), n, d, self._ptr(out))
        return out

    def scores(self, v, variant: int = L2) -> np.ndarray:
        v = self._u16(v)
        n, d = v.shape
        out = np.empty(n, np.float64)
        self.lib.vdo_scores(self._ptr(v), n, d, int(variant), self._ptr(out))
        return out

    def scores_weighted(self, v, a, variant: int = L2) -> np.ndarray:
        """App. A Eq. (app_fastcaote): a_j / (1 - a_j) * s_j."""
        v = self._u16(v)
        n, d = v.shape
        a = np.ascontiguousarray(a, dtype=np.float64)
        out = np.empty(n, np.float64)
        self.lib.vdo_scores_weighted(self._ptr(v), n, d, int(variant), self._ptr(a), self._ptr(out))
        return out

    def dispersion(self, x) -> float:
        """Sec. 3.1: std over tokens of ||x_i - mean|| (population)."""
        x = self._u16(x)
        n, d = x.shape
        return float(self.lib.vdo_dispersion(self._ptr(x), n, d))

    # -- Eq. (eviction) ---------------------------------------------------
    def select_top_n(self, scores, N: int) -> np.ndarray:
        s = np.ascontiguousarray(scores, dtype=np.float64)
        n = s.shape[0]
        kept = np.empty(min(n, N), np.int32)
        m = self.lib.vdo_select_top_n(self._ptr(s), n, int(N), self._ptr(kept))
        return kept[:m]

    def evict_unit(self, k, v, N: int, variant: int = L2):
        """Returns (k', v', kept, scores-or-None); k' and v' hold min(n, N) rows."""
        k = self._u16(k).copy()
        v = self._u16(v).copy()
        n, d = v.shape
        kept = np.empty(min(n, N), np.int32)
        s = np.empty(n, np.float64)
        m = self.lib.vdo_evict_unit(self._ptr(k), self._ptr(v), n, d, int(N), int(variant),
                                    self._ptr(kept), self._ptr(s))
        return k[:m], v[:m], kept[:m], (s if n > N else None)

    def evict_units(self, k, v, len_per_seq, N_per_seq, units_per_seq: int,
                    variant: int = L2, nthreads: int = 1, kept_stride: int = 0):
        """In place on k, v shaped [U, capacity, d] (uint16).  Returns kept
        [U, kept_stride] (-1 past each unit's kept count) when kept_stride > 0."""
        assert k.flags.c_contiguous and v.flags.c_contiguous
        assert k.dtype == np.uint16 and v.dtype == np.uint16
        U, cap, d = v.shape
        ln = np.ascontiguousarray(len_per_seq, np.int32)
        Ns = np.ascontiguousarray(N_per_seq, np.int32)
        kept = None
        if kept_stride:
            kept = np.full((U, kept_stride), -1, np.int32)
        rc = self.lib.vdo_evict_units(self._ptr(k), self._ptr(v), self._ptr(ln), self._ptr(Ns),
                                      U, int(units_per_seq), cap, d, int(variant),
                                      self._ptr(kept) if kept is not None else None,
                                      int(kept_stride), int(nthreads))
        if rc != 0:
            raise RuntimeError("oracle worker threads could not be started")
        return kept

    # -- Eq. (block_processing) -------------------------------------------
    def block_process(self, k_stream, v_stream, B: int, N: int, variant: int = L2):
        """Sec. 2.2: C_i <- pi_N([C_{i-1} || block_i]) for every block of B
        tokens of a [T, d] stream (the last block may be shorter).  Returns the
        final (k, v) cache and, per block, the kept indices of that event
        (None where the cache did not exceed N)."""
        k_stream = self._u16(k_stream)
        v_stream = self._u16(v_stream)
        T, d = v_stream.shape
        kc = np.empty((0, d), np.uint16)
        vc = np.empty((0, d), np.uint16)
        events = []
        for start in range(0, T, B):
            kc = np.concatenate([kc, k_stream[start:start + B]])
            vc = np.concatenate([vc, v_stream[start:start + B]])
            if vc.shape[0] > N:
                kc, vc, kept, _ = self.evict_unit(kc, vc, N, variant)
                events.append(kept)
            else:
                events.append(None)
        return kc, vc, events


def load(path: str | None = None) -> Oracle:
    """The oracle compiled from this directory (built on first use)."""
    global _lib
    if path is not None:
        return Oracle(path)
    with _lock:
        if _lib is None:
            _lib = Oracle(build())
        return _lib


def bf16_bits(x) -> np.ndarray:
    """Round float values to bf16 (nearest-even) and return the bit patterns.
    For building small test inputs; exact for small integers."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    w = f.view(np.uint32).astype(np.uint64)
    rounding = ((w >> 16) & 1) + 0x7FFF
    out = ((w + rounding) >> 16).astype(np.uint16)
    nan = np.isnan(f)
    out[nan] = 0x7FC0
    return out


def bits_to_float(b) -> np.ndarray:
    """bf16 bit patterns -> float64 (exact)."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
