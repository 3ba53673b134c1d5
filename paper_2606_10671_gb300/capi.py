"""ctypes declarations of the C ABI in include/fademem.h (same names, same arguments).

Argument marshalling only: every step of the method runs in libfademem.so.
Loading fails loudly when the library is missing; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfademem.so")

FADEMEM_OK = 0
FADEMEM_ERR_INVALID_ARG = 1
FADEMEM_ERR_UNSUPPORTED = 2
FADEMEM_ERR_WORKSPACE = 3
FADEMEM_ERR_EMPTY = 4
FADEMEM_ERR_PENDING = 5
FADEMEM_ERR_CUDA = 6
FADEMEM_ERR_DEVICE_TIMEOUT = 7
FADEMEM_ERR_DEVICE_CHECK = 8
# Bits of the device status word (include/fademem.h, FADEMEM_STATUS_*).
STATUS_TIMEOUT = 0x1
STATUS_COUNT_MISMATCH = 0x2
STATUS_PLAN_OVERFLOW = 0x4
STATUS_NEAR_TIE = 0x8
STATUS_BOUNDS = 0x10
# Bits of fademem_build_flags() (FADEMEM_BUILD_*).
BUILD_DEBUG_BOUNDS = 0x1
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "WORKSPACE", 4: "EMPTY", 5: "PENDING", 6: "CUDA",
                7: "DEVICE_TIMEOUT", 8: "DEVICE_CHECK"}

FADEMEM_F32, FADEMEM_BF16 = 0, 1
FADEMEM_MERGE_WEIGHTED, FADEMEM_MERGE_AVERAGE, FADEMEM_MERGE_SELECT_NEAREST, FADEMEM_MERGE_MAX_POOL = 0, 1, 2, 3
FADEMEM_MAX_BUDGET = 64
FADEMEM_MAX_LAYERS = 128
FADEMEM_MAX_PENDING = 64

# Every symbol include/fademem.h declares.
EXPORTS = ("fademem_workspace_bytes", "fademem_create", "fademem_insert", "fademem_consolidate", "fademem_attend",
           "fademem_attend_ext",
           "fademem_counts", "fademem_get_entries", "fademem_last_plan", "fademem_stats",
           "fademem_layer_memory", "fademem_get_device_status",
           "fademem_selftest_wait_timeout", "fademem_reset", "fademem_consolidate_noalloc",
           "fademem_host_staging_bytes", "fademem_step_host", "fademem_state_bytes", "fademem_export_state",
           "fademem_import_state", "fademem_destroy", "fademem_build_flags", "fademem_last_error")


class fademem_config(ctypes.Structure):
    _fields_ = [("budget", ctypes.c_int), ("heads", ctypes.c_int), ("head_dim", ctypes.c_int),
                ("tokens_per_frame", ctypes.c_int), ("num_layers", ctypes.c_int), ("beta", ctypes.c_double),
                ("anchor", ctypes.c_int), ("merge_op", ctypes.c_int), ("dtype", ctypes.c_int),
                ("scale", ctypes.c_float), ("rope_pairs", ctypes.c_int), ("rope_theta", ctypes.c_double)]


class FadeMemError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


_lock = threading.Lock()
_lib = None


def load(path: str | None = None):
    """Load libfademem.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"{p} is missing: run paper_2606_10671_gb300.build.build_library() "
                               "(the CUDA library is required; there is no CPU fallback)")
        lib = ctypes.CDLL(p)
        P, I, I64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
        cfgp = ctypes.POINTER(fademem_config)
        sig = {
            "fademem_workspace_bytes": (ctypes.c_size_t, [cfgp]),
            "fademem_create": (I, [cfgp, P, ctypes.c_size_t, ctypes.POINTER(P)]),
            "fademem_insert": (I, [P, I, P, P, I]),
            "fademem_consolidate": (I, [P, P]),
            "fademem_attend": (I, [P, I, P, P, I, P]),
            "fademem_attend_ext": (I, [P, I, P, P, P, I, P, I, P]),
            "fademem_counts": (I, [P, ctypes.POINTER(I), ctypes.POINTER(I64)]),
            "fademem_get_entries": (I, [P, P, I, ctypes.POINTER(I), P, P, P, P]),
            "fademem_last_plan": (I, [P, P, ctypes.POINTER(I), ctypes.POINTER(I), ctypes.POINTER(I)]),
            "fademem_stats": (I, [P, P, ctypes.POINTER(ctypes.c_uint64), ctypes.POINTER(ctypes.c_uint64),
                                  ctypes.POINTER(ctypes.c_uint64)]),
            "fademem_layer_memory": (I, [P, I, ctypes.POINTER(P), ctypes.POINTER(P)]),
            "fademem_get_device_status": (I, [P, P, ctypes.POINTER(ctypes.c_uint32)]),
            "fademem_selftest_wait_timeout": (I, [P, P]),
            "fademem_reset": (I, [P, P]),
            "fademem_consolidate_noalloc": (I, [P, P]),
            "fademem_host_staging_bytes": (ctypes.c_size_t, [cfgp, I, I]),
            "fademem_step_host": (I, [P, ctypes.POINTER(P), ctypes.POINTER(P), I, I, P, P, I, P, ctypes.c_size_t, P]),
            "fademem_state_bytes": (ctypes.c_size_t, [P]),
            "fademem_export_state": (I, [P, P, ctypes.c_size_t, P]),
            "fademem_import_state": (I, [P, P, ctypes.c_size_t, P]),
            "fademem_destroy": (None, [P]),
            "fademem_build_flags": (ctypes.c_uint32, []),
            "fademem_last_error": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def check(status: int):
    if status != FADEMEM_OK:
        msg = load().fademem_last_error()
        raise FadeMemError(status, msg.decode() if msg else "")
    return status


# Thin wrappers with the C names (pointers as Python ints).
def fademem_workspace_bytes(cfg: fademem_config) -> int:
    return int(load().fademem_workspace_bytes(ctypes.byref(cfg)))


def fademem_create(cfg: fademem_config, workspace: int, nbytes: int) -> int:
    h = ctypes.c_void_p()
    check(load().fademem_create(ctypes.byref(cfg), ctypes.c_void_p(workspace), nbytes, ctypes.byref(h)))
    return h.value


def fademem_insert(h: int, layer: int, K: int, V: int, nframes: int):
    check(load().fademem_insert(ctypes.c_void_p(h), layer, ctypes.c_void_p(K), ctypes.c_void_p(V), nframes))


def fademem_consolidate(h: int, stream: int = 0):
    check(load().fademem_consolidate(ctypes.c_void_p(h), ctypes.c_void_p(stream)))


def fademem_attend(h: int, layer: int, Q: int, out: int, Lq: int, stream: int = 0):
    check(load().fademem_attend(ctypes.c_void_p(h), layer, ctypes.c_void_p(Q), ctypes.c_void_p(out), Lq,
                                ctypes.c_void_p(stream)))


def fademem_attend_ext(h: int, layer: int, Q: int, Kcur: int, Vcur: int, ncur: int, out: int, Lq: int,
                       stream: int = 0):
    check(load().fademem_attend_ext(ctypes.c_void_p(h), layer, ctypes.c_void_p(Q), ctypes.c_void_p(Kcur),
                                    ctypes.c_void_p(Vcur), ncur, ctypes.c_void_p(out), Lq, ctypes.c_void_p(stream)))


def fademem_counts(h: int):
    c, f = ctypes.c_int(), ctypes.c_int64()
    check(load().fademem_counts(ctypes.c_void_p(h), ctypes.byref(c), ctypes.byref(f)))
    return c.value, f.value


def fademem_get_entries(h: int, stream: int = 0, capacity: int = FADEMEM_MAX_BUDGET + 1):
    import numpy as np
    slot = np.zeros(capacity, np.int32)
    first = np.zeros(capacity, np.int64)
    span = np.zeros(capacity, np.int64)
    mu2 = np.zeros(capacity, np.int64)
    n = ctypes.c_int()
    check(load().fademem_get_entries(ctypes.c_void_p(h), ctypes.c_void_p(stream), capacity, ctypes.byref(n),
                                     slot.ctypes.data, first.ctypes.data, span.ctypes.data, mu2.ctypes.data))
    k = n.value
    return slot[:k], first[:k], span[:k], mu2[:k]


def fademem_last_plan(h: int, stream: int = 0):
    ns, nd, nf = ctypes.c_int(), ctypes.c_int(), ctypes.c_int()
    check(load().fademem_last_plan(ctypes.c_void_p(h), ctypes.c_void_p(stream), ctypes.byref(ns), ctypes.byref(nd),
                                   ctypes.byref(nf)))
    return ns.value, nd.value, nf.value


def fademem_stats(h: int, stream: int = 0):
    b, n, k = ctypes.c_uint64(), ctypes.c_uint64(), ctypes.c_uint64()
    check(load().fademem_stats(ctypes.c_void_p(h), ctypes.c_void_p(stream), ctypes.byref(b), ctypes.byref(n),
                               ctypes.byref(k)))
    return b.value, n.value, k.value


def fademem_layer_memory(h: int, layer: int):
    k, v = ctypes.c_void_p(), ctypes.c_void_p()
    check(load().fademem_layer_memory(ctypes.c_void_p(h), layer, ctypes.byref(k), ctypes.byref(v)))
    return k.value, v.value


def fademem_get_device_status(h: int, stream: int = 0, raise_on_error: bool = True):
    w = ctypes.c_uint32()
    st = load().fademem_get_device_status(ctypes.c_void_p(h), ctypes.c_void_p(stream), ctypes.byref(w))
    if raise_on_error:
        check(st)
    return st, w.value


def fademem_selftest_wait_timeout(h: int, stream: int = 0):
    check(load().fademem_selftest_wait_timeout(ctypes.c_void_p(h), ctypes.c_void_p(stream)))


def fademem_reset(h: int, stream: int = 0):
    check(load().fademem_reset(ctypes.c_void_p(h), ctypes.c_void_p(stream)))


def fademem_consolidate_noalloc(h: int, stream: int = 0):
    check(load().fademem_consolidate_noalloc(ctypes.c_void_p(h), ctypes.c_void_p(stream)))


def fademem_host_staging_bytes(cfg: fademem_config, nframes: int, Lq: int) -> int:
    return int(load().fademem_host_staging_bytes(ctypes.byref(cfg), nframes, Lq))


def fademem_step_host(h: int, K_host, V_host, nframes: int, layer: int, Q_host: int, out_host: int, Lq: int,
                      staging: int, staging_bytes: int, stream: int = 0):
    """K_host, V_host: sequences of host addresses, one per layer."""
    n = len(K_host)
    Ks = (ctypes.c_void_p * n)(*K_host)
    Vs = (ctypes.c_void_p * n)(*V_host)
    check(load().fademem_step_host(ctypes.c_void_p(h), Ks, Vs, nframes, layer, ctypes.c_void_p(Q_host),
                                   ctypes.c_void_p(out_host), Lq, ctypes.c_void_p(staging), staging_bytes,
                                   ctypes.c_void_p(stream)))


def fademem_state_bytes(h: int) -> int:
    return int(load().fademem_state_bytes(ctypes.c_void_p(h)))


def fademem_export_state(h: int, stream: int = 0):
    """A snapshot of the memory as a numpy uint8 array."""
    import numpy as np
    buf = np.empty(fademem_state_bytes(h), np.uint8)
    check(load().fademem_export_state(ctypes.c_void_p(h), buf.ctypes.data, buf.size, ctypes.c_void_p(stream)))
    return buf


def fademem_import_state(h: int, snapshot, stream: int = 0):
    import numpy as np
    buf = np.ascontiguousarray(np.frombuffer(snapshot, np.uint8))
    check(load().fademem_import_state(ctypes.c_void_p(h), buf.ctypes.data, buf.size, ctypes.c_void_p(stream)))


def fademem_destroy(h: int):
    load().fademem_destroy(ctypes.c_void_p(h))


def fademem_build_flags() -> int:
    """FADEMEM_BUILD_* bits of the loaded library (BUILD_DEBUG_BOUNDS: the bounds-checking build)."""
    return int(load().fademem_build_flags())


def fademem_last_error() -> str:
    m = load().fademem_last_error()
    return m.decode() if m else ""
