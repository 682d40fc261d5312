"""The C ABI on its own: tests/c_abi/evict_example.c is a C program that
allocates with the CUDA runtime, calls libvd.so through include/vd.h only (no
Python or torch in its process), and checks a fused block event and a fused
decode step against the oracle's C code.  Building it needs no GPU; running
it needs a GB300."""
from __future__ import annotations

import os
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2609_23314_gb300")
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def build_example(out_dir) -> str:
    from paper_2609_23314_gb300 import build
    build.build()
    exe = os.path.join(str(out_dir), "evict_example")
    cmd = ["gcc", "-O2", "-std=c11", "-Wall", "-Werror", "-fno-fast-math", "-ffp-contract=off",
           os.path.join(ROOT, "tests", "c_abi", "evict_example.c"),
           os.path.join(ROOT, "oracle", "vd_oracle.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(ROOT, "oracle"),
           "-I", os.path.join(CUDA, "include"),
           "-L", PKG, "-lvd", "-L", os.path.join(CUDA, "lib64"), "-lcudart", "-lm", "-lpthread",
           f"-Wl,-rpath,{PKG}", f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}", "-o", exe]
    subprocess.run(cmd, check=True)
    return exe


def test_c_example_builds_against_the_header(tmp_path):
    assert os.access(build_example(tmp_path), os.X_OK)


@pytest.mark.gpu
def test_c_example_matches_the_oracle(tmp_path):
    exe = build_example(tmp_path)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "match the oracle" in r.stdout
