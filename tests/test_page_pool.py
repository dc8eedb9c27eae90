"""The host allocator of the paged KV cache (csrc/page_pool.h), on the CPU.

tests/page_pool_check.cpp is compiled with the host C++ compiler against the
same header the CUDA runtime includes. It checks the prefix-sharing, fork and
exhaustion scenarios and a seeded random walk against the pool's invariants:
reference counts, the free list and exact rollback.
"""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_page_pool_invariants(tmp_path):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path / "page_pool_check")
    subprocess.run([cxx, "-std=c++17", "-O1", "-Wall",
                    "-I", os.path.join(ROOT, "paper_2605_31464_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "page_pool_check.cpp"), "-o", exe], check=True)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == "ok"
