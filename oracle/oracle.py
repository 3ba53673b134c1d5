"""ctypes front end of the fp64 C oracle (test infrastructure only).

``build_oracle()`` compiles ``fademem_oracle.c`` with gcc into
``liboracle.so`` beside it; ``OracleMemory`` wraps one memory (one layer's
ordered entry list) and exposes Algorithm S1 one unit at a time plus the
brute-force attention over the memory.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

OP_WEIGHTED, OP_AVERAGE, OP_SELECT_NEAREST, OP_MAX_POOL = 0, 1, 2, 3

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fademem_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build_oracle(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP over query rows only)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        # FADEMEM_ORACLE_LIB: a separately built oracle (the sanitizer tests build one
        # with ASan/UBSan and run the pins against it).
        lib = ctypes.CDLL(os.environ.get("FADEMEM_ORACLE_LIB") or build_oracle())
        P = ctypes.c_void_p
        dp = ctypes.POINTER(ctypes.c_double)
        lib.oracle_create.restype = P
        lib.oracle_create.argtypes = [ctypes.c_int, ctypes.c_double, ctypes.c_int, ctypes.c_int,
                                      ctypes.c_longlong]
        lib.oracle_destroy.argtypes = [P]
        lib.oracle_insert.argtypes = [P, dp, dp]
        lib.oracle_count.argtypes = [P]
        lib.oracle_frames.argtypes = [P]
        lib.oracle_frames.restype = ctypes.c_longlong
        lib.oracle_last_pair.argtypes = [P]
        lib.oracle_last_margin.argtypes = [P]
        lib.oracle_last_margin.restype = ctypes.c_double
        lib.oracle_last_gmin.argtypes = [P]
        lib.oracle_last_gmin.restype = ctypes.c_double
        lib.oracle_entries.argtypes = [P, P, P, P, P]
        lib.oracle_entry_kv.argtypes = [P, ctypes.c_int, dp, dp]
        lib.oracle_attend.argtypes = [P, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp, ctypes.c_longlong,
                                      ctypes.c_double, dp]
        lib.oracle_attend_ext.argtypes = [P, ctypes.c_int, ctypes.c_int, ctypes.c_int, dp, dp, ctypes.c_longlong, dp,
                                          ctypes.c_longlong, ctypes.c_double, dp]
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_set_rope.argtypes = [P, ctypes.c_int, ctypes.c_double, ctypes.c_int, ctypes.c_int, ctypes.c_int]
        _lib = lib
        return lib


def oracle_num_threads() -> int:
    return int(_load().oracle_num_threads())


def _dptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_double))


class OracleMemory:
    """One FadeMem memory (Algorithm S1) in fp64.

    ``elems`` is the number of doubles in one K (or V) block; 0 runs the
    schedule alone.  For attention the block order is [tokens][heads][dim].
    """

    def __init__(self, budget: int, beta: float, anchor: bool = True, op: int = OP_WEIGHTED,
                 elems: int = 0):
        self._lib = _load()
        self.elems = int(elems)
        self._h = self._lib.oracle_create(int(budget), float(beta), int(bool(anchor)), int(op), self.elems)
        if not self._h:
            raise ValueError("oracle_create rejected its arguments")
        self.budget = int(budget)

    def set_rope(self, pairs: int, theta: float, tokens: int, heads: int, dim: int):
        """Temporal RoPE handling (before the first insert): keys are stored without their
        frame's phase and re-indexed at attention (see the C file's header)."""
        if self._lib.oracle_set_rope(self._h, int(pairs), float(theta), int(tokens), int(heads), int(dim)) != 0:
            raise ValueError("oracle_set_rope rejected its arguments")

    def close(self):
        if getattr(self, "_h", None):
            self._lib.oracle_destroy(self._h)
            self._h = None

    def __del__(self):
        self.close()

    def insert(self, K=None, V=None) -> int:
        """Algorithm S1 for one unit; returns the merged pair index j (-1: none)."""
        if self.elems:
            K = np.ascontiguousarray(K, dtype=np.float64).reshape(-1)
            V = np.ascontiguousarray(V, dtype=np.float64).reshape(-1)
            assert K.size == self.elems and V.size == self.elems
            self._lib.oracle_insert(self._h, _dptr(K), _dptr(V))
        else:
            self._lib.oracle_insert(self._h, None, None)
        return int(self._lib.oracle_last_pair(self._h))

    @property
    def count(self) -> int:
        return int(self._lib.oracle_count(self._h))

    @property
    def frames(self) -> int:
        return int(self._lib.oracle_frames(self._h))

    @property
    def last_margin(self) -> float:
        return float(self._lib.oracle_last_margin(self._h))

    @property
    def last_gmin(self) -> float:
        return float(self._lib.oracle_last_gmin(self._h))

    def entries(self):
        """(slot int32, first int64, span int64, mu float64) arrays, temporal order."""
        n = self.count
        slot = np.zeros(n, np.int32)
        first = np.zeros(n, np.int64)
        span = np.zeros(n, np.int64)
        mu = np.zeros(n, np.float64)
        self._lib.oracle_entries(self._h, slot.ctypes.data, first.ctypes.data, span.ctypes.data,
                                 mu.ctypes.data)
        return slot, first, span, mu

    def entry_kv(self, i: int):
        K = np.empty(self.elems, np.float64)
        V = np.empty(self.elems, np.float64)
        if self._lib.oracle_entry_kv(self._h, int(i), _dptr(K), _dptr(V)) != 0:
            raise IndexError(i)
        return K, V

    def attend(self, Q, tokens: int, heads: int, dim: int, scale: float | None = None) -> np.ndarray:
        """softmax(scale q K^T) V per head over every cached token; Q [Lq][heads][dim]."""
        Q = np.ascontiguousarray(Q, dtype=np.float64).reshape(-1, heads, dim)
        out = np.empty_like(Q)
        sc = 1.0 / np.sqrt(dim) if scale is None else float(scale)
        rc = self._lib.oracle_attend(self._h, int(tokens), int(heads), int(dim), _dptr(Q), Q.shape[0], sc,
                                     _dptr(out))
        if rc != 0:
            raise ValueError(f"oracle_attend failed ({rc})")
        return out

    def attend_ext(self, Q, Kcur, Vcur, tokens: int, heads: int, dim: int, scale: float | None = None) -> np.ndarray:
        """Attention over every cached token followed by the current chunk's tokens
        (Kcur, Vcur: [ncur][heads][dim], ncur may be 0)."""
        Q = np.ascontiguousarray(Q, dtype=np.float64).reshape(-1, heads, dim)
        Kc = np.ascontiguousarray(Kcur, dtype=np.float64).reshape(-1, heads, dim)
        Vc = np.ascontiguousarray(Vcur, dtype=np.float64).reshape(-1, heads, dim)
        assert Kc.shape == Vc.shape
        out = np.empty_like(Q)
        sc = 1.0 / np.sqrt(dim) if scale is None else float(scale)
        rc = self._lib.oracle_attend_ext(self._h, int(tokens), int(heads), int(dim), _dptr(Kc), _dptr(Vc), Kc.shape[0],
                                         _dptr(Q), Q.shape[0], sc, _dptr(out))
        if rc != 0:
            raise ValueError(f"oracle_attend_ext failed ({rc})")
        return out
