"""ctypes wrapper and builder for outer.c (test infrastructure only).

outer.c holds the two rank-one updates of the oracle's column sweep as plain
C loops over the rows (OpenMP), element by element the same operations as
numpy's outer product followed by a subtraction.  They make the literal
sweep (every compensation and every Schur downdate applied immediately to all
remaining columns) affordable at the widths of the large decoder blocks
(n = 4096 to 8192), where numpy's single-threaded temporaries take tens of
minutes.  Without a C compiler the numpy statement is used; both give the same
bits (tests/test_oracle_pins.py)."""
from __future__ import annotations

import ctypes
import os
import subprocess
from concurrent.futures import ThreadPoolExecutor

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "outer.c")
_LIB = os.path.join(_HERE, "libouter.so")
_lib = None
_failed = False


def build(force: bool = False) -> str:
    """Compile outer.c into oracle/libouter.so (OpenMP if the compiler has it)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        base = ["gcc", "-O2", "-ffp-contract=off", "-shared", "-fPIC", "-o", _LIB, _SRC]
        if subprocess.run(base[:3] + ["-fopenmp"] + base[3:], capture_output=True).returncode != 0:
            subprocess.check_call(base)
    return _LIB


def _load():
    global _lib, _failed
    if _lib is None and not _failed:
        try:
            build()
            lib = ctypes.CDLL(_LIB)
        except Exception:
            _failed = True
            return None
        dp = ctypes.POINTER(ctypes.c_double)
        i64 = ctypes.c_int64
        lib.realq_oracle_outer_sub.argtypes = [i64, i64, dp, i64, dp, i64, dp]
        lib.realq_oracle_outer_sub.restype = None
        lib.realq_oracle_outer_sub_div.argtypes = [i64, i64, dp, i64, dp, i64, dp, ctypes.c_double]
        lib.realq_oracle_outer_sub_div.restype = None
        _lib = lib
    return _lib


def _view(a: np.ndarray):
    """(pointer, leading stride in elements) of a 2-D fp64 view with unit inner stride, or None."""
    if a.dtype != np.float64 or a.ndim != 2 or (a.shape[1] > 1 and a.strides[1] != 8) or a.strides[0] % 8:
        return None
    return ctypes.cast(a.ctypes.data, ctypes.POINTER(ctypes.c_double)), a.strides[0] // 8


def _vec(u: np.ndarray):
    if u.dtype != np.float64 or u.ndim != 1 or (u.shape[0] > 1 and u.strides[0] % 8):
        return None
    return ctypes.cast(u.ctypes.data, ctypes.POINTER(ctypes.c_double)), (u.strides[0] // 8 if u.shape[0] > 1 else 1)


def outer_sub(A: np.ndarray, u: np.ndarray, v: np.ndarray, d: float = None) -> None:
    """In place: A -= np.outer(u, v) (d None) or A -= np.outer(u, v) / d."""
    rows, cols = A.shape
    if rows == 0 or cols == 0:
        return
    lib = _load()
    av, uv = _view(A), _vec(u)
    vc = np.ascontiguousarray(v, dtype=np.float64)
    if lib is None or av is None or uv is None or v.dtype != np.float64:
        if d is None:
            A -= np.outer(u, v)
        else:
            A -= np.outer(u, v) / d
        return
    vp = ctypes.cast(vc.ctypes.data, ctypes.POINTER(ctypes.c_double))
    if d is None:
        lib.realq_oracle_outer_sub(rows, cols, av[0], av[1], uv[0], uv[1], vp)
    else:
        lib.realq_oracle_outer_sub_div(rows, cols, av[0], av[1], uv[0], uv[1], vp, float(d))


_pool = None


def row_chunks(rows: int, size: int, fn, min_size: int = 1 << 20) -> None:
    """fn(r0, r1) over row ranges covering [0, rows): in one call for small
    work, else split among threads (numpy releases the interpreter lock in
    its elementwise loops).  The ranges do not overlap."""
    global _pool
    nt = os.cpu_count() or 1
    if size < min_size or nt == 1 or rows < 2:
        fn(0, rows)
        return
    if _pool is None:
        _pool = ThreadPoolExecutor(nt)
    step = -(-rows // nt)
    futs = [_pool.submit(fn, r0, min(rows, r0 + step)) for r0 in range(0, rows, step)]
    for f in futs:
        f.result()
