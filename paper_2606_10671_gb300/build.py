"""Build libfademem.so in-tree with nvcc for sm_103a (no GPU needed to build).

Each translation unit under csrc/ compiles in parallel to an object in
_build/, then nvcc links them with the static CUDA runtime, so the library
loads on a machine without a driver (for the symbol checks) and needs no
libcudart at run time.  A source hash skips rebuilds when nothing changed.

`--debug-bounds` (build_library(debug_bounds=True)) builds
libfademem_debug.so instead, with -DFADEMEM_DEBUG_BOUNDS: every kernel then
checks each global-memory access and table index and reports a failure
through the device status word (FADEMEM_STATUS_BOUNDS) rather than making it.
"""
from __future__ import annotations

import concurrent.futures as cf
import hashlib
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "libfademem.so")
LIB_DEBUG = os.path.join(HERE, "libfademem_debug.so")
DEBUG_FLAGS = ["-DFADEMEM_DEBUG_BOUNDS"]
INCLUDE = os.path.join(ROOT, "include")
SOURCES = ["fademem_api.cu", "consolidate.cu", "attend_simt.cu", "attend_tc.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden", "-I", INCLUDE]


def _nvcc() -> str:
    cand = os.environ.get("NVCC") or shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(cand) and shutil.which(cand) is None:
        raise RuntimeError("nvcc not found: the FadeMem CUDA library cannot be built")
    return cand


def _digest(extra: list[str]) -> str:
    h = hashlib.sha256()
    files = sorted(os.listdir(CSRC)) + ["../../include/fademem.h", "../build.py"]
    for name in files:
        path = os.path.normpath(os.path.join(CSRC, name))
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as fh:
                h.update(fh.read())
    # The flags without the include directory's absolute path, so that the same sources
    # give the same digest on every machine.
    h.update(" ".join(ARCH + [f for f in NVCC_FLAGS if f != INCLUDE] + extra).encode())
    return h.hexdigest()


def build_library(force: bool = False, verbose: bool = False, debug_bounds: bool = False) -> str:
    """Compile (if stale) and return the path of libfademem.so (libfademem_debug.so
    with device bounds checks when debug_bounds)."""
    extra = DEBUG_FLAGS if debug_bounds else []
    out = LIB_DEBUG if debug_bounds else LIB
    build = os.path.join(BUILD, "debug") if debug_bounds else BUILD
    stamp = os.path.join(build, "stamp")
    digest = _digest(extra)
    if not force and os.path.exists(out) and os.path.exists(stamp):
        with open(stamp) as fh:
            if fh.read().strip() == digest:
                return out
    os.makedirs(build, exist_ok=True)
    nvcc = _nvcc()

    def compile_one(src: str) -> str:
        obj = os.path.join(build, src.replace(".cu", ".o"))
        cmd = [nvcc, *ARCH, *NVCC_FLAGS, *extra, "-c", os.path.join(CSRC, src), "-o", obj]
        if verbose:
            cmd.insert(1, "-Xptxas=-v")
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode != 0:
            raise RuntimeError(f"nvcc failed on {src}:\n{r.stdout}\n{r.stderr}")
        if verbose and (r.stdout or r.stderr):
            sys.stderr.write(r.stdout + r.stderr)
        return obj

    with cf.ThreadPoolExecutor(max_workers=len(SOURCES)) as ex:
        objs = list(ex.map(compile_one, SOURCES))
    tmp = out + f".tmp{os.getpid()}"
    cmd = [nvcc, *ARCH, "-shared", "-cudart", "static", "-o", tmp, *objs, "-ldl"]  # -ldl: NVTX loads its tool lazily
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(f"nvcc link failed:\n{r.stdout}\n{r.stderr}")
    os.replace(tmp, out)
    with open(stamp, "w") as fh:
        fh.write(digest)
    return out


if __name__ == "__main__":
    print(build_library(force="--force" in sys.argv, verbose="-v" in sys.argv,
                        debug_bounds="--debug-bounds" in sys.argv))
