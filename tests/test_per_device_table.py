"""The library keeps device properties and per-device settings (multiprocessor
count, the attention kernel's shared-memory opt-in, the no-alloc scratch
address) in a per-device table (csrc/per_device.h), so a process that drives
several GPUs launches correctly on each.  Its logic has no CUDA dependency and
is checked here on the host: built with g++ (threads included) and run."""
import os
import shutil
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.skipif(shutil.which("g++") is None, reason="needs g++")
def test_per_device_table(tmp_path):
    exe = tmp_path / "per_device_table_check"
    subprocess.run(["g++", "-std=c++17", "-O1", "-pthread", "-Wall", "-Werror",
                    "-I", os.path.join(ROOT, "paper_2606_10671_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "per_device_table_check.cpp"), "-o", str(exe)], check=True)
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0 and r.stdout.strip() == "ok", r.stdout + r.stderr

