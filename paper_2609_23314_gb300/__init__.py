"""GB300 (sm_103a) ValueDiff KV-cache eviction: Python binding of libvd.so.

A thin ctypes layer over the C ABI in ``include/vd.h``, with the same names.
It only marshals arguments -- torch tensors in, device pointers and the
caller's CUDA stream out -- and checks dtypes, devices and shapes so that no
wrong pointer reaches the library.  Every step of the eviction runs in the
CUDA kernels of ``csrc/``; there is no CPU or PyTorch fallback: if
``libvd.so`` has not been built, every call raises.

The method (paper: ValueDiff, Sec. 3.2 Eq. vd; Sec. 2.1 Eq. eviction;
Sec. 2.2 Eq. block_processing): per (sequence, layer, KV head), score each
cached token by ||v_j - mean(V)||_2 (or the Dir / Norm variants), keep the N
highest scores (ties to the lower slot) and compact K and V in place.
"""
from __future__ import annotations

import ctypes
import os
import threading

__all__ = [
    "VD_SCORE_L2", "VD_SCORE_DIR", "VD_SCORE_NORM", "VD_MU_RECOMPUTE", "VD_MU_RUNNING",
    "VdError", "Cache", "vd_score", "vd_score_ex", "vd_evict_block", "vd_evict_block_ex",
    "vd_append_evict_block", "vd_append_evict_block_ex", "vd_append_evict_decode",
    "vd_evict_decode",
    "vd_evict_block_holefill", "vd_evict_decode_holefill", "vd_append",
    "vd_running_sum_init", "vd_running_sum_init_ex", "vd_workspace_size", "vd_status_string",
    "vd_get_device_status",
    "library_path", "load_library",
]

VD_SCORE_L2, VD_SCORE_DIR, VD_SCORE_NORM = 0, 1, 2
VD_MU_RECOMPUTE, VD_MU_RUNNING = 0, 1
VARIANTS = {"l2": VD_SCORE_L2, "dir": VD_SCORE_DIR, "norm": VD_SCORE_NORM}

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libvd.so")
_lib = None
_lock = threading.Lock()


class VdError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = int(code)
        super().__init__(f"{where}: {vd_status_string(code)} (status {code})")


class _VdCache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("len", ctypes.c_void_p),
                ("n_seq", ctypes.c_int32), ("n_layer", ctypes.c_int32),
                ("n_kv_head", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("capacity", ctypes.c_int32)]


def library_path() -> str:
    return _LIB_PATH


def load_library() -> ctypes.CDLL:
    """Load the in-tree libvd.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB_PATH):
                raise RuntimeError(f"{_LIB_PATH} is missing: build it with "
                                   "paper_2609_23314_gb300.build.build() (nvcc, sm_103a)")
            lib = ctypes.CDLL(_LIB_PATH)
            P, I32, S = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int
            cp = ctypes.POINTER(_VdCache)
            lib.vd_score.argtypes = [cp, S, P, P]
            lib.vd_evict_block.argtypes = [cp, I32, P, I32, S, S, P, P, P, P]
            lib.vd_append_evict_block.argtypes = [cp, P, P, I32, I32, P, S, S, P, P, P, P, P, P]
            lib.vd_append_evict_decode.argtypes = [cp, P, P, I32, P, S, S, P, P, P, P, P, P, P]
            lib.vd_evict_decode.argtypes = [cp, I32, P, S, S, P, P, P, P, P]
            lib.vd_evict_block_holefill.argtypes = [cp, I32, P, I32, S, S, P, P, P, P, P, P]
            lib.vd_evict_decode_holefill.argtypes = [cp, I32, P, S, S, P, P, P, P, P, P, P]
            lib.vd_score_ex.argtypes = [cp, S, S, P, I32, P, P, P]
            lib.vd_evict_block_ex.argtypes = [cp, I32, P, I32, S, S, P, I32, P, P, P, P, P]
            lib.vd_append_evict_block_ex.argtypes = [cp, P, P, I32, I32, P, S, S, P, I32, P, P, P,
                                                     P, P]
            lib.vd_append.argtypes = [cp, P, P, I32, P]
            lib.vd_running_sum_init.argtypes = [cp, P, P]
            lib.vd_running_sum_init_ex.argtypes = [cp, I32, P, P]
            lib.vd_workspace_size.argtypes = [cp]
            lib.vd_workspace_size.restype = ctypes.c_size_t
            lib.vd_status_string.argtypes = [S]
            lib.vd_status_string.restype = ctypes.c_char_p
            lib.vd_get_device_status.argtypes = [P]
            for f in ("vd_score", "vd_score_ex", "vd_evict_block_ex", "vd_evict_block",
                      "vd_append_evict_block", "vd_append_evict_block_ex", "vd_append_evict_decode",
                      "vd_evict_decode", "vd_evict_block_holefill",
                      "vd_evict_decode_holefill", "vd_append", "vd_running_sum_init",
                      "vd_running_sum_init_ex",
                      "vd_get_device_status"):
                getattr(lib, f).restype = S
            _lib = lib
        return _lib


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------
def _torch():
    import torch
    return torch


def _stream(stream):
    if stream is None:
        return ctypes.c_void_p(_torch().cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _ptr(t, dtype, shape, what, device):
    """The tensor's device pointer after checking its type, device, layout
    and shape (so that no wrong pointer reaches the library)."""
    if t is None:
        return None
    try:
        ok = (t.dtype == dtype and t.get_device() == (device.index if device.type == "cuda" else -1)
              and t.is_contiguous() and t.shape == shape)
    except AttributeError:
        raise TypeError(f"{what} must be a torch tensor") from None
    if not ok:
        if t.dtype != dtype:
            raise TypeError(f"{what} must be {dtype}, got {t.dtype}")
        if t.device != device:
            raise ValueError(f"{what} must live on {device}, got {t.device}")
        if not t.is_contiguous():
            raise ValueError(f"{what} must be contiguous")
        raise ValueError(f"{what} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    return t.data_ptr()


def _check(code: int, where: str):
    if code != 0:
        raise VdError(code, where)


class Cache:
    """A KV cache in the library's layout: K and V bf16
    [n_seq, n_layer, n_kv_head, capacity, head_dim] and len int32 [n_seq],
    all on one CUDA device.  Holds references to the tensors only."""

    def __init__(self, k, v, len):
        torch = _torch()
        if k.dim() != 5 or k.shape != v.shape:
            raise ValueError("k and v must both be [n_seq, n_layer, n_kv_head, capacity, head_dim]")
        self.k, self.v, self.len = k, v, len
        self.n_seq, self.n_layer, self.n_kv_head, self.capacity, self.head_dim = (int(x) for x in k.shape)
        self.device = k.device
        _ptr(k, torch.bfloat16, k.shape, "k", self.device)
        _ptr(v, torch.bfloat16, k.shape, "v", self.device)
        _ptr(len, torch.int32, (self.n_seq,), "len", self.device)
        self._s = _VdCache(k.data_ptr(), v.data_ptr(), len.data_ptr(), self.n_seq, self.n_layer,
                           self.n_kv_head, self.head_dim, self.capacity)

    @classmethod
    def empty(cls, n_seq, n_layer, n_kv_head, capacity, head_dim, device="cuda"):
        torch = _torch()
        shape = (n_seq, n_layer, n_kv_head, capacity, head_dim)
        return cls(torch.zeros(shape, dtype=torch.bfloat16, device=device),
                   torch.zeros(shape, dtype=torch.bfloat16, device=device),
                   torch.zeros(n_seq, dtype=torch.int32, device=device))

    @property
    def units(self) -> int:
        return self.n_seq * self.n_layer * self.n_kv_head

    def unit_shape(self):
        return (self.n_seq, self.n_layer, self.n_kv_head)

    def ref(self):
        return ctypes.byref(self._s)


# ---------------------------------------------------------------------------
# the C ABI, same names
# ---------------------------------------------------------------------------
def vd_score(cache: Cache, variant: int, scores_out, stream=None) -> None:
    torch = _torch()
    sc = _ptr(scores_out, torch.float32, cache.unit_shape() + (cache.capacity,), "scores_out", cache.device)
    _check(load_library().vd_score(cache.ref(), int(variant), sc, _stream(stream)), "vd_score")


def vd_evict_block(cache: Cache, N: int, N_dev=None, B: int = 0, variant: int = VD_SCORE_L2,
                   mu: int = VD_MU_RECOMPUTE, running_sum=None, kept_idx_out=None,
                   scores_out=None, stream=None) -> None:
    torch = _torch()
    us = cache.unit_shape()
    args = (
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
    )
    _check(load_library().vd_evict_block(cache.ref(), int(N), args[0], int(B), int(variant), int(mu),
                                         args[1], args[2], args[3], _stream(stream)),
           "vd_evict_block")


def vd_append_evict_block(cache: Cache, k_new, v_new, B: int, N: int, N_dev=None,
                          variant: int = VD_SCORE_L2, mu: int = VD_MU_RECOMPUTE,
                          running_sum=None, kept_idx_out=None, scores_out=None,
                          stream=None, pos=None, pos_first_new=None) -> None:
    """vd_append followed by vd_evict_block (or, with pos and pos_first_new,
    vd_evict_block_holefill) in one launch; k_new, v_new: bf16
    [n_seq, n_layer, n_kv_head, B, head_dim], read straight from the caller's
    buffers (only surviving rows are written into the cache)."""
    torch = _torch()
    us = cache.unit_shape()
    shape = us + (int(B), cache.head_dim)
    args = (
        _ptr(k_new, torch.bfloat16, shape, "k_new", cache.device),
        _ptr(v_new, torch.bfloat16, shape, "v_new", cache.device),
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
        _ptr(pos, torch.int32, us + (cache.capacity,), "pos", cache.device),
        _ptr(pos_first_new, torch.int32, (cache.n_seq,), "pos_first_new", cache.device),
    )
    _check(load_library().vd_append_evict_block(cache.ref(), args[0], args[1], int(B), int(N),
                                                args[2], int(variant), int(mu), args[3],
                                                args[6], args[7], args[4], args[5],
                                                _stream(stream)),
           "vd_append_evict_block")


def vd_append_evict_decode(cache: Cache, k_new, v_new, N: int, N_dev=None,
                           variant: int = VD_SCORE_L2, mu: int = VD_MU_RECOMPUTE,
                           running_sum=None, evicted_out=None, kept_idx_out=None,
                           scores_out=None, stream=None, pos=None, pos_first_new=None) -> None:
    """vd_append of one token followed by vd_evict_decode (or, with pos and
    pos_first_new, vd_evict_decode_holefill) in one launch; k_new, v_new:
    bf16 [n_seq, n_layer, n_kv_head, 1, head_dim]."""
    torch = _torch()
    us = cache.unit_shape()
    shape = us + (1, cache.head_dim)
    args = (
        _ptr(k_new, torch.bfloat16, shape, "k_new", cache.device),
        _ptr(v_new, torch.bfloat16, shape, "v_new", cache.device),
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(pos, torch.int32, us + (cache.capacity,), "pos", cache.device),
        _ptr(pos_first_new, torch.int32, (cache.n_seq,), "pos_first_new", cache.device),
        _ptr(evicted_out, torch.int32, us, "evicted_out", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
    )
    _check(load_library().vd_append_evict_decode(cache.ref(), args[0], args[1], int(N), args[2],
                                                 int(variant), int(mu), args[3], args[4],
                                                 args[5], args[6], args[7], args[8],
                                                 _stream(stream)),
           "vd_append_evict_decode")


def vd_evict_decode(cache: Cache, N: int, N_dev=None, variant: int = VD_SCORE_L2,
                    mu: int = VD_MU_RECOMPUTE, running_sum=None, evicted_out=None,
                    kept_idx_out=None, scores_out=None, stream=None) -> None:
    torch = _torch()
    us = cache.unit_shape()
    args = (
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(evicted_out, torch.int32, us, "evicted_out", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
    )
    _check(load_library().vd_evict_decode(cache.ref(), int(N), args[0], int(variant), int(mu),
                                          args[1], args[2], args[3], args[4], _stream(stream)),
           "vd_evict_decode")


def vd_score_ex(cache: Cache, variant: int, score_keys: bool = False, scores_out=None,
                dispersion_out=None, stream=None, mu: int = VD_MU_RECOMPUTE,
                running_sum=None) -> None:
    """Scores of V (or K) rows and/or the per-unit dispersion sigma; with
    mu=VD_MU_RUNNING the mean is running_sum / len (fp64 [n_seq, n_layer,
    n_kv_head, head_dim], read only), so the rows are read once."""
    torch = _torch()
    us = cache.unit_shape()
    sc = _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device)
    dp = _ptr(dispersion_out, torch.float32, us, "dispersion_out", cache.device)
    rs = _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device)
    _check(load_library().vd_score_ex(cache.ref(), int(variant), int(mu), rs,
                                      int(bool(score_keys)), sc, dp, _stream(stream)),
           "vd_score_ex")


def vd_evict_block_ex(cache: Cache, N: int, N_dev=None, B: int = 0, variant: int = VD_SCORE_L2,
                      mu: int = VD_MU_RECOMPUTE, running_sum=None, score_keys: bool = False,
                      attn=None, kept_idx_out=None, scores_out=None, dispersion_out=None,
                      stream=None) -> None:
    """Block eviction on the K-side rule and/or with attention weights;
    dispersion_out: fp32 [n_seq, n_layer, n_kv_head], sigma of the
    pre-eviction rows from the same score pass (units that evicted)."""
    torch = _torch()
    us = cache.unit_shape()
    args = (
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(attn, torch.float32, us + (cache.capacity,), "attn", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
        _ptr(dispersion_out, torch.float32, us, "dispersion_out", cache.device),
    )
    _check(load_library().vd_evict_block_ex(cache.ref(), int(N), args[0], int(B), int(variant),
                                            int(mu), args[1], int(bool(score_keys)), args[2],
                                            args[3], args[4], args[5], _stream(stream)),
           "vd_evict_block_ex")


def vd_append_evict_block_ex(cache: Cache, k_new, v_new, B: int, N: int, N_dev=None,
                             variant: int = VD_SCORE_L2, mu: int = VD_MU_RECOMPUTE,
                             running_sum=None, score_keys: bool = False, attn=None,
                             kept_idx_out=None, scores_out=None, dispersion_out=None,
                             stream=None) -> None:
    """vd_append followed by vd_evict_block_ex in one launch; k_new, v_new:
    bf16 [n_seq, n_layer, n_kv_head, B, head_dim], read straight from the
    caller's buffers (attn covers the new rows at slots len .. len + B - 1)."""
    torch = _torch()
    us = cache.unit_shape()
    shape = us + (int(B), cache.head_dim)
    args = (
        _ptr(k_new, torch.bfloat16, shape, "k_new", cache.device),
        _ptr(v_new, torch.bfloat16, shape, "v_new", cache.device),
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(attn, torch.float32, us + (cache.capacity,), "attn", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
        _ptr(dispersion_out, torch.float32, us, "dispersion_out", cache.device),
    )
    _check(load_library().vd_append_evict_block_ex(
        cache.ref(), args[0], args[1], int(B), int(N), args[2], int(variant), int(mu), args[3],
        int(bool(score_keys)), args[4], args[5], args[6], args[7], _stream(stream)),
        "vd_append_evict_block_ex")


def vd_evict_block_holefill(cache: Cache, N: int, pos, pos_first_new, N_dev=None, B: int = 0,
                            variant: int = VD_SCORE_L2, mu: int = VD_MU_RECOMPUTE,
                            running_sum=None, kept_idx_out=None, scores_out=None,
                            stream=None) -> None:
    """Block eviction in the hole-fill layout (kept appended rows move into the
    evicted slots; ties by token position).  pos: int32 [.., capacity]
    positions of the cached rows; pos_first_new: int32 [n_seq]."""
    torch = _torch()
    us = cache.unit_shape()
    args = (
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(pos, torch.int32, us + (cache.capacity,), "pos", cache.device),
        _ptr(pos_first_new, torch.int32, (cache.n_seq,), "pos_first_new", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
    )
    _check(load_library().vd_evict_block_holefill(cache.ref(), int(N), args[0], int(B), int(variant),
                                                  int(mu), args[1], args[2], args[3], args[4],
                                                  args[5], _stream(stream)),
           "vd_evict_block_holefill")


def vd_evict_decode_holefill(cache: Cache, N: int, pos, pos_first_new, N_dev=None,
                             variant: int = VD_SCORE_L2, mu: int = VD_MU_RECOMPUTE,
                             running_sum=None, evicted_out=None, kept_idx_out=None,
                             scores_out=None, stream=None) -> None:
    """Decode eviction in the hole-fill layout: the appended token moves into
    the evicted slot (at most one row moves)."""
    torch = _torch()
    us = cache.unit_shape()
    args = (
        _ptr(N_dev, torch.int32, (cache.n_seq,), "N_dev", cache.device),
        _ptr(running_sum, torch.float64, us + (cache.head_dim,), "running_sum", cache.device),
        _ptr(pos, torch.int32, us + (cache.capacity,), "pos", cache.device),
        _ptr(pos_first_new, torch.int32, (cache.n_seq,), "pos_first_new", cache.device),
        _ptr(evicted_out, torch.int32, us, "evicted_out", cache.device),
        _ptr(kept_idx_out, torch.int32, us + (int(N),), "kept_idx_out", cache.device),
        _ptr(scores_out, torch.float32, us + (cache.capacity,), "scores_out", cache.device),
    )
    _check(load_library().vd_evict_decode_holefill(cache.ref(), int(N), args[0], int(variant),
                                                   int(mu), args[1], args[2], args[3], args[4],
                                                   args[5], args[6], _stream(stream)),
           "vd_evict_decode_holefill")


def vd_append(cache: Cache, k_new, v_new, B: int, stream=None) -> None:
    torch = _torch()
    shape = cache.unit_shape() + (int(B), cache.head_dim)
    kp = _ptr(k_new, torch.bfloat16, shape, "k_new", cache.device)
    vp = _ptr(v_new, torch.bfloat16, shape, "v_new", cache.device)
    _check(load_library().vd_append(cache.ref(), kp, vp, int(B), _stream(stream)), "vd_append")


def vd_running_sum_init_ex(cache: Cache, of_keys: bool, running_sum, stream=None) -> None:
    """fp64 column sums of the cached K rows (of_keys) or V rows, per unit."""
    torch = _torch()
    rp = _ptr(running_sum, torch.float64, cache.unit_shape() + (cache.head_dim,), "running_sum",
              cache.device)
    _check(load_library().vd_running_sum_init_ex(cache.ref(), int(bool(of_keys)), rp,
                                                 _stream(stream)), "vd_running_sum_init_ex")


def vd_running_sum_init(cache: Cache, running_sum, stream=None) -> None:
    torch = _torch()
    rp = _ptr(running_sum, torch.float64, cache.unit_shape() + (cache.head_dim,), "running_sum",
              cache.device)
    _check(load_library().vd_running_sum_init(cache.ref(), rp, _stream(stream)), "vd_running_sum_init")


def vd_workspace_size(cache: Cache) -> int:
    return int(load_library().vd_workspace_size(cache.ref()))


def vd_status_string(code: int) -> str:
    return load_library().vd_status_string(int(code)).decode()


def vd_get_device_status(stream=None) -> int:
    """Synchronises the stream and returns (and clears) the device status."""
    return int(load_library().vd_get_device_status(_stream(stream)))
