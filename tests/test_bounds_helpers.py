"""The range test of the bounds-checking build (csrc/fademem_internal.h, range_holds)
pinned on the host: built with g++ against the CUDA headers and run (no GPU needed).
Every kernel check of libfademem_debug.so goes through it."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA_INCLUDE = "/usr/local/cuda/include"


@pytest.mark.skipif(shutil.which("g++") is None or not os.path.isdir(CUDA_INCLUDE), reason="needs g++ and CUDA headers")
def test_range_holds(tmp_path):
    exe = tmp_path / "bounds_helpers_check"
    subprocess.run(["g++", "-std=c++17", "-O1", "-Wall", "-Werror", "-I", CUDA_INCLUDE,
                    "-I", os.path.join(ROOT, "paper_2606_10671_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "bounds_helpers_check.cpp"), "-o", str(exe)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr
