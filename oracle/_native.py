"""Builds and loads the oracle's C brute-force searcher (oracle/brute.c). Test infrastructure only."""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "brute.c")
_LIB = os.path.join(_HERE, "_brute.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile brute.c with the host C compiler into oracle/_brute.so."""
    stale = (not os.path.exists(_LIB)) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-shared", "-fPIC", "-o", tmp, _SRC])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        f = lib.lcvq_oracle_brute_nearest
        f.restype = ctypes.c_int
        f.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64, ctypes.c_int,
                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p]
        _lib = lib
    return _lib


def brute_nearest(W, A, b, d: int):
    W64 = np.ascontiguousarray(W, dtype=np.float64)
    A64 = np.ascontiguousarray(A, dtype=np.float64)
    b64 = np.ascontiguousarray(b, dtype=np.float64)
    m, n = W64.shape
    codes = np.zeros((m, n), dtype=np.uint8)
    dist = np.zeros((m, n // d), dtype=np.float64)
    rc = _load().lcvq_oracle_brute_nearest(W64.ctypes.data, m, n, d, A64.ctypes.data, b64.ctypes.data,
                                           codes.ctypes.data, dist.ctypes.data)
    if rc != 0:
        raise ValueError("brute_nearest: bad arguments")
    return codes, dist
