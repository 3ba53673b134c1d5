"""The GPU parity cases again, through the bounds-checking build (GPU only).

libfademem_debug.so (build.py --debug-bounds) compiles every kernel with
FADEMEM_DEBUG_BOUNDS: each global-memory access is checked against the buffer
it belongs to (the workspace's memory slabs, the caller's frames, queries and
outputs) and each table index against its array; an access that fails is
skipped and recorded as FADEMEM_STATUS_BOUNDS in the device status word, which
the parity helpers read after every check of the entry table and the tests at
their end, and which must stay clear.  This runs every test
of test_gpu_parity.py, test_gpu_configs.py and test_gpu_attend_split.py in a
subprocess that loads that build: the seeded fuzz over every option, every
consolidation kernel instance, RoPE, the current chunk, multi-layer memories up
to 128 layers, the fp32 path, the full Wan-1.3B shapes, CUDA graphs,
checkpoints, the attention's slow paths and its cluster split, the hour-long
stress, the 30-layer rollout and the 40-layer Wan-14B memory.
They must pass unchanged, with the status word clear.
"""
import ctypes
import os
import subprocess
import sys

import pytest
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="needs a CUDA GPU")]


def test_parity_cases_under_bounds_checks():
    from paper_2606_10671_gb300 import build, capi
    debug = build.build_library(debug_bounds=True)
    lib = ctypes.CDLL(debug)
    lib.fademem_build_flags.restype = ctypes.c_uint32
    assert lib.fademem_build_flags() == capi.BUILD_DEBUG_BOUNDS
    env = dict(os.environ, FADEMEM_CUDA_LIB=debug)
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider", "-m", "gpu",
                        os.path.join(HERE, "test_gpu_parity.py"), os.path.join(HERE, "test_gpu_configs.py"),
                        os.path.join(HERE, "test_gpu_attend_split.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=1500)
    tail = r.stdout[-3000:] + r.stderr[-2000:]
    assert r.returncode == 0, tail
    assert " passed" in r.stdout and " failed" not in r.stdout, tail
    print(r.stdout.strip().splitlines()[-1])
