"""The C ABI used from plain C (tests/c_abi_consumer.c): compiled with gcc against
include/fademem.h, linked with libfademem.so, the CUDA runtime and the fp64 oracle."""
import os
import subprocess

import pytest
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _compile(out, cuda_lib, oracle_lib):
    libdir = os.path.dirname(cuda_lib)
    odir = os.path.dirname(oracle_lib)
    cmd = ["gcc", "-std=c11", "-O2", "-Wall", "-o", out, os.path.join(HERE, "c_abi_consumer.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
           cuda_lib, oracle_lib, "-L", os.path.join(CUDA, "lib64"), "-lcudart", "-lm",
           f"-Wl,-rpath,{libdir}:{odir}:{os.path.join(CUDA, 'lib64')}"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)


def test_c_consumer_compiles(cuda_lib, oracle_lib, tmp_path):
    """The header is valid C11 and every declared symbol resolves at link time."""
    _compile(str(tmp_path / "consumer"), cuda_lib, oracle_lib)


@pytest.mark.gpu
@pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")
def test_c_consumer_runs(cuda_lib, oracle_lib, tmp_path):
    exe = str(tmp_path / "consumer")
    _compile(exe, cuda_lib, oracle_lib)
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stdout + r.stderr
    assert "ok" in r.stdout
