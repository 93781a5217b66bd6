"""Python access to ``column_reduce.c``: the plain, multi-threaded CPU Allreduce by its
definition (every rank ends with the op-reduction of all P inputs; Sec.
"Introduction").

TEST INFRASTRUCTURE, NOT PRODUCT CODE (see ``oracle/__init__.py``).  Used as the
multi-threaded CPU baseline of ``bench.py`` and, in ``tests/``, as a second
implementation of the definition for the cases where the result does not depend on
the association order (int32 wraparound sums, max, min).
"""

from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "column_reduce.c")
_LIB = os.path.join(_HERE, "libcolumn_reduce.so")
_DT = {"f32": (0, np.float32), "i32": (2, np.int32)}
_OPS = {"sum": 0, "max": 1, "min": 2}
_lib = None


def build(force: bool = False) -> str:
    """Compiles column_reduce.c with the system C compiler (portable C + pthreads)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-O3", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", tmp, _SRC],
                       check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(build())
        _lib.column_allreduce.restype = ctypes.c_int
        _lib.column_allreduce.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                          ctypes.c_size_t, ctypes.c_int, ctypes.c_int, ctypes.c_int]
    return _lib


def column_allreduce_ptrs(in_ptrs, out_ptrs, n: int, dtype: str, op: str, threads: int) -> None:
    """Runs on P input and P output addresses (host memory, n elements each)."""
    P = len(in_ptrs)
    a = (ctypes.c_void_p * P)(*in_ptrs)
    b = (ctypes.c_void_p * P)(*out_ptrs)
    rc = _load().column_allreduce(a, b, P, n, _DT[dtype][0], _OPS[op], threads)
    if rc != 0:
        raise ValueError("column_allreduce: bad argument")


def column_allreduce(inputs, op: str = "sum", dtype: str = "f32", threads: int = 1):
    """Returns the P output vectors (all equal) for P input vectors."""
    want = _DT[dtype][1]
    xs = [np.ascontiguousarray(v, dtype=want) for v in inputs]
    n = len(xs[0]) if xs else 0
    outs = [np.empty(n, want) for _ in xs]
    column_allreduce_ptrs([v.ctypes.data for v in xs], [o.ctypes.data for o in outs], n, dtype, op,
                          threads)
    return outs
