"""libvd.so loads and exports every entry point include/vd.h declares; host
validation rejects bad arguments before touching the GPU (CPU only)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "vd.h")


def declared_functions():
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(vd_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_23314_gb300 import build, load_library
    build.build()
    return load_library()


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("vd_score", "vd_evict_block", "vd_evict_decode", "vd_append",
                     "vd_running_sum_init", "vd_workspace_size", "vd_status_string",
                     "vd_get_device_status"):
        assert required in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in vd.h but not exported by libvd.so"


def test_status_strings(lib):
    for code in range(0, 12):
        s = lib.vd_status_string(code)
        assert isinstance(s, bytes) and len(s) > 0
    assert lib.vd_status_string(0) == b"ok"


def _cache(k=0x1000, v=0x2000, ln=0x3000, n_seq=1, n_layer=2, n_kv_head=2, head_dim=64,
           capacity=128):
    from paper_2609_23314_gb300 import _VdCache
    return _VdCache(k, v, ln, n_seq, n_layer, n_kv_head, head_dim, capacity)


def test_workspace_size_is_zero(lib):
    c = _cache()
    assert lib.vd_workspace_size(ctypes.byref(c)) == 0


@pytest.mark.parametrize("fields,code", [
    (dict(head_dim=12), 2),          # not a multiple of 8
    (dict(head_dim=264), 3),         # wider than the kernels handle
    (dict(k=0x1008), 2),             # K not 16-byte aligned
    (dict(v=0), 1),                  # null V
    (dict(ln=0), 1),                 # null len
    (dict(n_layer=0), 1),
    (dict(capacity=0), 1),
])
def test_bad_cache_rejected_before_launch(lib, fields, code):
    c = _cache(**fields)
    rc = lib.vd_evict_block(ctypes.byref(c), 16, None, 4, 0, 0, None, None, None, None)
    assert rc == code


def test_bad_arguments_rejected_before_launch(lib):
    c = _cache()
    ref = ctypes.byref(c)
    assert lib.vd_evict_block(None, 16, None, 4, 0, 0, None, None, None, None) == 1
    assert lib.vd_evict_block(ref, 0, None, 4, 0, 0, None, None, None, None) == 1      # N < 1
    assert lib.vd_evict_block(ref, 129, None, 4, 0, 0, None, None, None, None) == 1    # N > capacity
    assert lib.vd_evict_block(ref, 16, None, -1, 0, 0, None, None, None, None) == 1    # B < 0
    assert lib.vd_evict_block(ref, 16, None, 4, 7, 0, None, None, None, None) == 1     # variant
    assert lib.vd_evict_block(ref, 16, None, 4, 0, 1, None, None, None, None) == 1     # running, no sum
    assert lib.vd_evict_decode(ref, 16, None, 0, 3, None, None, None, None, None) == 1  # mu mode
    assert lib.vd_score(ref, 0, None, None) == 1                                      # no output
    assert lib.vd_append(ref, None, None, 4, None) == 1
    assert lib.vd_append(ref, 0x18, 0x28, 4, None) == 2                               # unaligned rows
    assert lib.vd_running_sum_init(ref, None, None) == 1


def test_scoring_options_rejected_before_launch(lib):
    c = _cache()
    ref = ctypes.byref(c)
    sigma = 0x40
    # sigma is defined on the L2 distance
    assert lib.vd_evict_block_ex(ref, 16, None, 4, 1, 0, None, 0, None, None, None, sigma,
                                 None) == 1
    assert lib.vd_score_ex(ref, 2, 0, None, 0, None, sigma, None) == 1
    assert lib.vd_score_ex(ref, 0, 0, None, 0, None, None, None) == 1        # no output
    assert lib.vd_score_ex(ref, 0, 1, None, 0, None, sigma, None) == 1       # running, no sum
    assert lib.vd_score_ex(ref, 0, 5, None, 0, None, sigma, None) == 1       # unknown mean mode
    # the running mean needs its sum, for either tensor
    assert lib.vd_evict_block_ex(ref, 16, None, 4, 0, 1, None, 1, None, None, None, None,
                                 None) == 1
    assert lib.vd_running_sum_init_ex(ref, 1, None, None) == 1
    # fused append: both buffers, B >= 1, 16-byte aligned
    assert lib.vd_append_evict_block(ref, 0x100, 0x200, 0, 16, None, 0, 0, None, None, None,
                                     None, None, None) == 1
    assert lib.vd_append_evict_block(ref, 0x100, None, 4, 16, None, 0, 0, None, None, None,
                                     None, None, None) == 1
    assert lib.vd_append_evict_block(ref, 0x108, 0x200, 4, 16, None, 0, 0, None, None, None,
                                     None, None, None) == 2
    assert lib.vd_append_evict_block(ref, 0x100, 0x200, 4, 16, None, 0, 0, None, 0x300, None,
                                     None, None, None) == 1            # one position array
    # the fused form of the scoring options: the same checks as both halves
    assert lib.vd_append_evict_block_ex(ref, 0x100, None, 4, 16, None, 0, 0, None, 0, None,
                                        None, None, None, None) == 1
    assert lib.vd_append_evict_block_ex(ref, 0x108, 0x200, 4, 16, None, 0, 0, None, 0, None,
                                        None, None, None, None) == 2
    assert lib.vd_append_evict_block_ex(ref, 0x100, 0x200, 4, 16, None, 1, 0, None, 0, None,
                                        None, None, 0x40, None) == 1   # sigma needs L2
    assert lib.vd_append_evict_block_ex(ref, 0x100, 0x200, 4, 16, None, 0, 1, None, 1, None,
                                        None, None, None, None) == 1   # running, no sum
    # the hole-fill layout needs both position arrays
    assert lib.vd_evict_block_holefill(ref, 16, None, 4, 0, 0, None, 0x40, None, None, None,
                                       None) == 1
    assert lib.vd_evict_decode_holefill(ref, 16, None, 0, 0, None, None, 0x40, None, None,
                                        None, None) == 1


def test_binding_checks_every_tensor_argument():
    """The binding passes a pointer only for a tensor of the expected dtype,
    device, shape and layout; anything else raises before the library is
    called."""
    import torch
    import paper_2609_23314_gb300 as vd
    cuda0 = torch.device("cuda", 0)
    cpu = torch.device("cpu")
    t = torch.zeros(2, 3, dtype=torch.float32)
    assert vd._ptr(None, torch.float32, (2, 3), "x", cpu) is None
    assert vd._ptr(t, torch.float32, (2, 3), "x", cpu) == t.data_ptr()
    with pytest.raises(TypeError):
        vd._ptr(t, torch.int32, (2, 3), "x", cpu)
    with pytest.raises(TypeError):
        vd._ptr([1, 2], torch.float32, (2,), "x", cpu)
    with pytest.raises(ValueError, match="live on"):
        vd._ptr(t, torch.float32, (2, 3), "x", cuda0)
    with pytest.raises(ValueError, match="contiguous"):
        vd._ptr(t.t(), torch.float32, (3, 2), "x", cpu)
    with pytest.raises(ValueError, match="shape"):
        vd._ptr(t, torch.float32, (3, 2), "x", cpu)
