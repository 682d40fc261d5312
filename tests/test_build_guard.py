"""The build's check on ptxas resource usage (CPU only): a kernel with a
local-memory stack frame or spills fails the build unless allowed."""
from paper_2609_23314_gb300 import build

LOG = """ptxas info    : Compiling entry function '_ZN2vd12evict_kernelILi0ELb1ELb0ELb1EEEvNS_9EvictArgsE' for 'sm_103a'
ptxas info    : Function properties for _ZN2vd12evict_kernelILi0ELb1ELb0ELb1EEEvNS_9EvictArgsE
    8 bytes stack frame, 4 bytes spill stores, 20 bytes spill loads
ptxas info    : Used 64 registers, used 1 barriers, 8 bytes cumulative stack size
ptxas info    : Compiling entry function '_Z17vd_len_add_kernelPiiii' for 'sm_103a'
ptxas info    : Function properties for _Z17vd_len_add_kernelPiiii
    0 bytes stack frame, 0 bytes spill stores, 0 bytes spill loads
ptxas info    : Used 8 registers, used 0 barriers
"""


def test_parse_resources():
    r = build.parse_resources(LOG)
    assert r["_ZN2vd12evict_kernelILi0ELb1ELb0ELb1EEEvNS_9EvictArgsE"] == (64, 8, 4, 20)
    assert r["_Z17vd_len_add_kernelPiiii"] == (8, 0, 0, 0)


def test_check_resources_flags_frames_not_allowed():
    r = build.parse_resources(LOG)
    k = "_ZN2vd12evict_kernelILi0ELb1ELb0ELb1EEEvNS_9EvictArgsE"
    assert build.check_resources(r) == [k]
    assert build.check_resources(r, allowed=frozenset({k})) == []
    assert build.ALLOWED_FRAMES == frozenset()
