"""Host-side code under AddressSanitizer and UndefinedBehaviorSanitizer (CPU only).

The fp64 oracle is rebuilt with -fsanitize=address,undefined (no recovery: any report
aborts) and its pins run against that build in a subprocess with the ASan runtime
preloaded.
"""
import os
import shutil
import subprocess
import sys

import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SAN = ["-fsanitize=address,undefined", "-fno-sanitize-recover=all", "-fno-omit-frame-pointer", "-g", "-O1"]


def _runtime(name):
    path = subprocess.run(["gcc", f"-print-file-name={name}"], capture_output=True, text=True).stdout.strip()
    return path if os.path.isabs(path) and os.path.exists(path) else None


@pytest.mark.skipif(shutil.which("gcc") is None, reason="needs gcc")
def test_oracle_pins_under_asan_ubsan(tmp_path):
    asan = _runtime("libasan.so")
    if asan is None:
        pytest.skip("no ASan runtime for this gcc")
    lib = str(tmp_path / "liboracle_san.so")
    subprocess.run(["gcc", *SAN, "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", lib,
                    os.path.join(ROOT, "oracle", "fademem_oracle.c"), "-lm"], check=True)
    env = dict(os.environ, FADEMEM_ORACLE_LIB=lib, LD_PRELOAD=asan,
               ASAN_OPTIONS="detect_leaks=0:abort_on_error=1", UBSAN_OPTIONS="halt_on_error=1:print_stacktrace=1",
               OMP_NUM_THREADS="2")
    sel = "golden or invariant or closed_form or properties or attention or rope or rejects"
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(HERE, "test_oracle_pins.py"), "-k", sel],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "passed" in r.stdout


@pytest.mark.skipif(shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"),
                    reason="needs nvcc")
def test_abi_host_code_under_asan_ubsan(tmp_path):
    """The library's host code (argument checks, workspace and staging sizing, snapshot
    header checks, the no-GPU error path) built with ASan/UBSan, driven by the CPU ABI tests."""
    asan = _runtime("libasan.so")
    if asan is None:
        pytest.skip("no ASan runtime for this gcc")
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    csrc = os.path.join(ROOT, "paper_2606_10671_gb300", "csrc")
    host_san = "-fPIC,-fvisibility=hidden,-fsanitize=address,-fsanitize=undefined,-fno-sanitize-recover=all," \
               "-fno-omit-frame-pointer"
    objs, procs = [], []
    for src in ("fademem_api", "consolidate", "attend_simt", "attend_tc"):
        obj = str(tmp_path / f"{src}.o")
        objs.append(obj)
        procs.append(subprocess.Popen([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O1", "-std=c++17",
                                       "-Xcompiler", host_san, "-I", os.path.join(ROOT, "include"), "-c",
                                       os.path.join(csrc, f"{src}.cu"), "-o", obj]))
    assert all(p.wait() == 0 for p in procs)
    lib = str(tmp_path / "libfademem_san.so")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-shared", "-cudart", "static",
                    "-Xcompiler", "-fsanitize=address,-fsanitize=undefined", "-o", lib, *objs, "-ldl"], check=True)
    env = dict(os.environ, FADEMEM_CUDA_LIB=lib, LD_PRELOAD=asan,
               ASAN_OPTIONS="detect_leaks=0:abort_on_error=1:protect_shadow_gap=0", UBSAN_OPTIONS="halt_on_error=1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", "-m", "not gpu",
                        os.path.join(HERE, "test_abi_cpu.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert "passed" in r.stdout
