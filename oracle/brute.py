"""ctypes wrapper and builder for brute.c (test infrastructure only)."""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "brute.c")
_LIB = os.path.join(_HERE, "libbrute.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile brute.c into oracle/libbrute.so with the host C compiler."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        subprocess.check_call(["gcc", "-O2", "-shared", "-fPIC", "-o", _LIB, _SRC])
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        dp = ctypes.POINTER(ctypes.c_double)
        ip = ctypes.POINTER(ctypes.c_int32)
        lib.realq_brute_row_min.argtypes = [ctypes.c_int, ctypes.c_int, dp, dp, ip]
        lib.realq_brute_row_min.restype = ctypes.c_double
        lib.realq_brute_row_eval.argtypes = [ctypes.c_int, ctypes.c_int, dp, dp, ip]
        lib.realq_brute_row_eval.restype = ctypes.c_double
        _lib = lib
    return _lib


def _ptr(a, t):
    return a.ctypes.data_as(ctypes.POINTER(t))


def _deltas(w0_row, scale, zero, levels):
    c = np.arange(levels, dtype=np.float32)
    grid = (np.float32(scale) * (c - np.float32(zero))).astype(np.float64)
    return np.ascontiguousarray(grid[None, :] - np.asarray(w0_row, dtype=np.float64)[:, None])


def row_min(w0_row, scale, zero, H, levels=16):
    """(min over all codes of delta^T H delta, argmin codes) for one row."""
    lib = _load()
    n = len(w0_row)
    H = np.ascontiguousarray(H, dtype=np.float64)
    dv = _deltas(w0_row, scale, zero, levels)
    arg = np.zeros(n, dtype=np.int32)
    best = lib.realq_brute_row_min(n, levels, _ptr(H, ctypes.c_double), _ptr(dv, ctypes.c_double),
                                   _ptr(arg, ctypes.c_int32))
    return best, arg.astype(np.int64)


def row_eval(w0_row, scale, zero, H, codes, levels=16):
    lib = _load()
    n = len(w0_row)
    H = np.ascontiguousarray(H, dtype=np.float64)
    dv = _deltas(w0_row, scale, zero, levels)
    c = np.ascontiguousarray(codes, dtype=np.int32)
    return lib.realq_brute_row_eval(n, levels, _ptr(H, ctypes.c_double), _ptr(dv, ctypes.c_double),
                                    _ptr(c, ctypes.c_int32))


def layer_min(W0, scales, zeros, H, levels=16, threads=4):
    """Row-wise brute force over a whole (tiny) layer; rows run in parallel threads."""
    m = W0.shape[0]
    with ThreadPoolExecutor(threads) as ex:
        res = list(ex.map(lambda i: row_min(W0[i], scales[i], zeros[i], H, levels), range(m)))
    return np.array([r[0] for r in res]), np.stack([r[1] for r in res])
