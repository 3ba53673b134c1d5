"""C ABI checks that need no GPU: the library builds and loads, exports every
symbol include/fademem.h declares, and validates arguments on the host (every
error returns a status and a message; nothing aborts)."""
import ctypes
import os
import re

import pytest
import torch

from paper_2606_10671_gb300 import capi, make_config

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FAKE_WS = 1 << 40  # 256-aligned address; host-only calls never dereference it


def _declared_symbols():
    hdr = open(os.path.join(ROOT, "include", "fademem.h")).read()
    return sorted(set(re.findall(r"FADEMEM_API[^;(]*?\b(fademem_\w+)\s*\(", hdr)))


def test_exports_every_declared_symbol(cuda_lib):
    lib = ctypes.CDLL(cuda_lib)
    declared = _declared_symbols()
    assert len(declared) == 23
    for name in declared:
        assert hasattr(lib, name), name
    assert sorted(capi.EXPORTS) == declared


def test_only_abi_symbols_exported(cuda_lib):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", cuda_lib], capture_output=True, text=True).stdout
    text = [ln.split()[-1] for ln in out.splitlines() if " T " in ln]
    assert sorted(text) == _declared_symbols()


def test_build_flags(cuda_lib):
    """The release library reports no build flags.  The bounds-checking build (nvcc,
    -DFADEMEM_DEBUG_BOUNDS; compiled here, no GPU needed) reports FADEMEM_BUILD_DEBUG_BOUNDS
    and exports exactly the same symbols."""
    import subprocess
    from paper_2606_10671_gb300 import build
    if not os.environ.get("FADEMEM_CUDA_LIB"):
        assert ctypes.CDLL(cuda_lib).fademem_build_flags() == 0
    debug = build.build_library(debug_bounds=True)
    lib = ctypes.CDLL(debug)
    lib.fademem_build_flags.restype = ctypes.c_uint32
    assert lib.fademem_build_flags() == capi.BUILD_DEBUG_BOUNDS
    out = subprocess.run(["nm", "-D", "--defined-only", debug], capture_output=True, text=True).stdout
    assert sorted(ln.split()[-1] for ln in out.splitlines() if " T " in ln) == _declared_symbols()


def _cfg(**kw):
    base = dict(budget=21, heads=12, head_dim=128, tokens_per_frame=1560, num_layers=1, beta=0.3, anchor=True,
                merge_op="weighted", dtype=torch.bfloat16)
    base.update(kw)
    return make_config(**base)


def test_workspace_bytes(cuda_lib):
    capi.load(cuda_lib)
    n = capi.fademem_workspace_bytes(_cfg())
    kv = 12 * 21 * 1560 * 128 * 2 * 2  # K and V of one layer, bf16
    assert kv <= n < kv + 64 * 1024
    n3 = capi.fademem_workspace_bytes(_cfg(num_layers=3))
    assert n3 - n == 2 * (kv + (-kv % 256))
    n32 = capi.fademem_workspace_bytes(_cfg(dtype=torch.float32))
    assert n32 - n == kv
    for bad in (dict(budget=1), dict(budget=65), dict(heads=0), dict(head_dim=96), dict(tokens_per_frame=0),
                dict(num_layers=0), dict(num_layers=129), dict(beta=0.0), dict(beta=1.5), dict(head_dim=64),
                dict(rope_pairs=-1), dict(rope_pairs=65), dict(rope_pairs=4, rope_theta=0.5)):
        assert capi.fademem_workspace_bytes(_cfg(**bad)) == 0, bad
    # Temporal RoPE adds the attention keys: a third [H][M][N][D] block per layer.
    nr = capi.fademem_workspace_bytes(_cfg(rope_pairs=22))
    assert nr - n == kv // 2 + (-(kv + kv // 2) % 256) - (-kv % 256)
    assert capi.fademem_workspace_bytes(_cfg(rope_pairs=64, rope_theta=500.0)) == nr


def _create_status(cfg, ws=FAKE_WS, nbytes=None):
    lib = capi.load()
    h = ctypes.c_void_p()
    if nbytes is None:
        nbytes = capi.fademem_workspace_bytes(cfg) or 1 << 30
    st = lib.fademem_create(ctypes.byref(cfg), ctypes.c_void_p(ws), nbytes, ctypes.byref(h))
    return st, h.value


def test_create_validation(cuda_lib):
    capi.load(cuda_lib)
    lib = capi.load()
    assert _create_status(_cfg(budget=1))[0] == capi.FADEMEM_ERR_INVALID_ARG
    assert "budget" in capi.fademem_last_error()
    assert _create_status(_cfg(beta=-1.0))[0] == capi.FADEMEM_ERR_INVALID_ARG
    assert _create_status(_cfg(head_dim=64))[0] == capi.FADEMEM_ERR_UNSUPPORTED
    assert _create_status(_cfg(), ws=0)[0] == capi.FADEMEM_ERR_WORKSPACE
    assert _create_status(_cfg(), ws=FAKE_WS + 16)[0] == capi.FADEMEM_ERR_WORKSPACE
    assert _create_status(_cfg(), nbytes=1024)[0] == capi.FADEMEM_ERR_WORKSPACE
    cfg = _cfg()
    assert lib.fademem_create(ctypes.byref(cfg), ctypes.c_void_p(FAKE_WS), 1 << 30, None) == \
        capi.FADEMEM_ERR_INVALID_ARG
    st, h = _create_status(_cfg(head_dim=64, dtype=torch.float32))
    assert st == capi.FADEMEM_OK and h
    capi.fademem_destroy(h)
    lib.fademem_destroy(None)  # NULL-safe


def test_host_side_call_checks(cuda_lib):
    """insert / attend / consolidate argument errors are caught before any CUDA call."""
    capi.load(cuda_lib)
    lib = capi.load()
    st, h = _create_status(_cfg(num_layers=2, tokens_per_frame=64, heads=2))
    assert st == capi.FADEMEM_OK
    H = ctypes.c_void_p(h)
    P = ctypes.c_void_p
    assert lib.fademem_insert(H, 2, P(FAKE_WS), P(FAKE_WS), 3) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_insert(H, -1, P(FAKE_WS), P(FAKE_WS), 3) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_insert(H, 0, None, P(FAKE_WS), 3) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_insert(H, 0, P(FAKE_WS + 8), P(FAKE_WS), 3) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_insert(H, 0, P(FAKE_WS), P(FAKE_WS), 0) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_attend(H, 0, P(FAKE_WS), P(FAKE_WS), 10, None) == capi.FADEMEM_ERR_EMPTY
    assert lib.fademem_insert(H, 0, P(FAKE_WS), P(FAKE_WS), 3) == capi.FADEMEM_OK
    assert lib.fademem_attend(H, 0, P(FAKE_WS), P(FAKE_WS), 10, None) == capi.FADEMEM_ERR_PENDING
    assert "consolidate" in capi.fademem_last_error()
    # layers disagree on their pending frames
    assert lib.fademem_consolidate(H, None) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_insert(H, 0, P(FAKE_WS), P(FAKE_WS), 62) == capi.FADEMEM_ERR_PENDING
    assert lib.fademem_attend(H, 5, P(FAKE_WS), P(FAKE_WS), 10, None) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_attend(H, 0, P(FAKE_WS), P(FAKE_WS), 0, None) == capi.FADEMEM_ERR_INVALID_ARG
    c, f = capi.fademem_counts(h)
    assert (c, f) == (0, 0)
    k, v = capi.fademem_layer_memory(h, 1)
    assert v - k == 2 * 21 * 64 * 128 * 2 and k > FAKE_WS
    capi.fademem_destroy(h)


def test_host_step_staging_and_checks(cuda_lib):
    """fademem_host_staging_bytes: two slots of (K, V per layer, Q, output), each piece
    256-byte aligned; fademem_step_host refuses bad arguments before any CUDA call."""
    capi.load(cuda_lib)
    lib = capi.load()
    r = lambda x: (x + 255) // 256 * 256
    cfg = _cfg(num_layers=2, tokens_per_frame=100, heads=3)
    frame = r(3 * 100 * 3 * 128 * 2)  # 3 frames of K (or V), bf16
    q = r(50 * 3 * 128 * 2)
    assert capi.fademem_host_staging_bytes(cfg, 3, 50) == 2 * (2 * 2 * frame + 2 * q)
    assert capi.fademem_host_staging_bytes(_cfg(dtype=torch.float32, num_layers=1, tokens_per_frame=7, heads=1), 1, 1) \
        == 2 * (2 * r(7 * 128 * 4) + 2 * r(128 * 4))
    for nf, lq in ((0, 50), (65, 50), (3, 0)):
        assert capi.fademem_host_staging_bytes(cfg, nf, lq) == 0
    assert capi.fademem_host_staging_bytes(_cfg(budget=1), 3, 50) == 0
    st, h = _create_status(cfg)
    assert st == capi.FADEMEM_OK
    P = ctypes.c_void_p
    need = capi.fademem_host_staging_bytes(cfg, 3, 50)
    host = (ctypes.c_char * 16)()
    hp = ctypes.addressof(host)
    two = (P * 2)(hp, hp)
    one_null = (P * 2)(hp, None)
    call = lambda K=two, V=two, nf=3, layer=0, Q=hp, out=hp, lq=50, stg=FAKE_WS, nb=need: lib.fademem_step_host(
        P(h), K, V, nf, layer, P(Q), P(out), lq, P(stg), nb, None)
    assert call(K=one_null) == capi.FADEMEM_ERR_INVALID_ARG
    assert call(Q=0) == capi.FADEMEM_ERR_INVALID_ARG
    assert call(layer=2) == capi.FADEMEM_ERR_INVALID_ARG
    assert call(nf=0) == capi.FADEMEM_ERR_INVALID_ARG
    assert call(nb=need - 1) == capi.FADEMEM_ERR_WORKSPACE
    assert "staging" in capi.fademem_last_error()
    assert call(stg=FAKE_WS + 8) == capi.FADEMEM_ERR_WORKSPACE
    assert call(stg=0) == capi.FADEMEM_ERR_WORKSPACE
    assert lib.fademem_step_host(None, two, two, 3, 0, P(hp), P(hp), 50, P(FAKE_WS), need, None) == \
        capi.FADEMEM_ERR_INVALID_ARG
    capi.fademem_destroy(h)


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU error path")
def test_cuda_failure_is_a_status(cuda_lib):
    """Without a GPU, the first device call returns FADEMEM_ERR_CUDA with the CUDA error text."""
    capi.load(cuda_lib)
    lib = capi.load()
    st, h = _create_status(_cfg(tokens_per_frame=16, heads=1))
    assert st == capi.FADEMEM_OK
    P = ctypes.c_void_p
    assert lib.fademem_insert(P(h), 0, P(FAKE_WS), P(FAKE_WS), 3) == capi.FADEMEM_OK
    assert lib.fademem_consolidate(P(h), None) == capi.FADEMEM_ERR_CUDA
    assert "cuda" in capi.fademem_last_error().lower()
    capi.fademem_destroy(h)


def test_snapshot_size_and_import_checks(cuda_lib):
    """fademem_state_bytes = header + entry table + K and V of every layer; imports of
    anything but a snapshot of the same configuration are refused before any CUDA call."""
    import struct
    capi.load(cuda_lib)
    lib = capi.load()
    cfg = _cfg(num_layers=2, tokens_per_frame=64, heads=2)
    st, h = _create_status(cfg)
    assert st == capi.FADEMEM_OK
    kv = 2 * 21 * 64 * 128 * 2  # one layer's K block: H*M*N*D bf16
    n = capi.fademem_state_bytes(h)
    overhead = n - 2 * 2 * kv
    assert 0 < overhead < 8192
    assert capi.fademem_state_bytes(None) == 0
    P = ctypes.c_void_p
    junk = (ctypes.c_char * n)()
    assert lib.fademem_import_state(P(h), junk, n, None) == capi.FADEMEM_ERR_INVALID_ARG
    assert "magic" in capi.fademem_last_error()
    assert lib.fademem_import_state(P(h), junk, 16, None) == capi.FADEMEM_ERR_INVALID_ARG
    # a header with the right magic and version but another configuration
    other = _cfg(num_layers=2, tokens_per_frame=64, heads=2, beta=0.5)
    hdr = b"FADEMEM\0" + struct.pack("<II", 1, 0) + bytes(other)
    buf = (ctypes.c_char * n).from_buffer_copy(hdr + b"\0" * (n - len(hdr)))
    st = lib.fademem_import_state(P(h), buf, n, None)
    assert st == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_export_state(P(h), None, n, None) == capi.FADEMEM_ERR_INVALID_ARG
    assert lib.fademem_export_state(P(h), junk, n - 1, None) == capi.FADEMEM_ERR_WORKSPACE
    capi.fademem_destroy(h)
