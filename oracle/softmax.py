"""ctypes front end of the double-precision softmax oracle (softmax_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline leg.  Arrays are numpy; bf16 data travels as uint16
bit patterns.  Nothing here touches the CUDA library.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

from . import build_oracle

F32 = 0
BF16 = 1
CAUSAL = 1

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = build_oracle.LIB
        if not os.path.exists(path):
            path = build_oracle.build()
        L = ctypes.CDLL(path)
        L.orc_softmax_row.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                      ctypes.c_int64, ctypes.c_uint32, ctypes.c_void_p,
                                      ctypes.c_void_p]
        L.orc_softmax_row.restype = ctypes.c_int
        L.orc_softmax_batched.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                          ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                          ctypes.c_uint32, ctypes.c_void_p, ctypes.c_void_p,
                                          ctypes.c_int]
        L.orc_softmax_batched.restype = ctypes.c_int
        L.orc_softmax_backward_row.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                               ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
        L.orc_softmax_backward_row.restype = ctypes.c_int
        L.orc_softmax_backward_batched.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int,
                                                   ctypes.c_int64, ctypes.c_void_p,
                                                   ctypes.c_void_p, ctypes.c_void_p,
                                                   ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int]
        L.orc_softmax_backward_batched.restype = ctypes.c_int
        L.orc_double_to_bf16.argtypes = [ctypes.c_double]
        L.orc_double_to_bf16.restype = ctypes.c_uint16
        _lib = L
    return _lib


def _dtype_code(x: np.ndarray) -> int:
    if x.dtype == np.float32:
        return F32
    if x.dtype == np.uint16:
        return BF16
    raise TypeError("oracle input must be float32 or uint16 (bf16 bits), got %s" % x.dtype)


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def softmax_row(xrow: np.ndarray, row_in_slice: int = 0, flags: int = 0):
    """Softmax of one row; returns (y as float64, y rounded to the input type)."""
    xrow = np.ascontiguousarray(xrow)
    dt = _dtype_code(xrow)
    C = xrow.shape[-1]
    y64 = np.empty(C, np.float64)
    yout = np.empty(C, xrow.dtype)
    rc = lib().orc_softmax_row(_ptr(xrow), dt, C, row_in_slice, flags, _ptr(y64), _ptr(yout))
    if rc:
        raise RuntimeError("orc_softmax_row failed: %d" % rc)
    return y64, yout


def softmax_batched(x: np.ndarray, offsets: Sequence[int], rows: Sequence[int],
                    cols: Sequence[int], flags: int = 0, want_f64: bool = True,
                    want_rounded: bool = True, nthreads: Optional[int] = None):
    """Softmax of every slice s (rows[s] x cols[s] elements at element offset
    offsets[s] of the flat array x).  Returns (y64 or None, yout or None), both
    the shape of x; elements outside every slice are left as NaN / 0."""
    x = np.ascontiguousarray(x).reshape(-1)
    dt = _dtype_code(x)
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    R = np.ascontiguousarray(rows, dtype=np.int32)
    C = np.ascontiguousarray(cols, dtype=np.int32)
    n = len(off)
    y64 = np.full(x.shape, np.nan, np.float64) if want_f64 else None
    yout = np.zeros(x.shape, x.dtype) if want_rounded else None
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    rc = lib().orc_softmax_batched(_ptr(x), dt, n, _ptr(off), _ptr(R), _ptr(C), flags,
                                   _ptr(y64), _ptr(yout), nthreads)
    if rc:
        raise RuntimeError("orc_softmax_batched failed: %d" % rc)
    return y64, yout


def softmax_backward_row(yrow: np.ndarray, dyrow: np.ndarray):
    """dx of one row (float64, rounded to the input type)."""
    yrow = np.ascontiguousarray(yrow)
    dyrow = np.ascontiguousarray(dyrow)
    dt = _dtype_code(yrow)
    assert dyrow.dtype == yrow.dtype and dyrow.shape == yrow.shape
    C = yrow.shape[-1]
    d64 = np.empty(C, np.float64)
    dout = np.empty(C, yrow.dtype)
    rc = lib().orc_softmax_backward_row(_ptr(yrow), _ptr(dyrow), dt, C, _ptr(d64), _ptr(dout))
    if rc:
        raise RuntimeError("orc_softmax_backward_row failed: %d" % rc)
    return d64, dout


def softmax_backward_batched(y: np.ndarray, dy: np.ndarray, offsets, rows, cols,
                             want_f64: bool = True, want_rounded: bool = True,
                             nthreads: Optional[int] = None):
    """dx = y * (dy - rowsum(y * dy)) for every slice; arrays flat, like x."""
    y = np.ascontiguousarray(y).reshape(-1)
    dy = np.ascontiguousarray(dy).reshape(-1)
    dt = _dtype_code(y)
    assert dy.dtype == y.dtype and dy.size == y.size
    off = np.ascontiguousarray(offsets, dtype=np.int64)
    R = np.ascontiguousarray(rows, dtype=np.int32)
    C = np.ascontiguousarray(cols, dtype=np.int32)
    d64 = np.full(y.shape, np.nan, np.float64) if want_f64 else None
    dout = np.zeros(y.shape, y.dtype) if want_rounded else None
    rc = lib().orc_softmax_backward_batched(_ptr(y), _ptr(dy), dt, len(off), _ptr(off), _ptr(R),
                                            _ptr(C), _ptr(d64), _ptr(dout),
                                            nthreads or os.cpu_count() or 1)
    if rc:
        raise RuntimeError("orc_softmax_backward_batched failed: %d" % rc)
    return d64, dout


def double_to_bf16(d: float) -> int:
    """The oracle's own round-to-nearest-even of a double to bf16 bits."""
    return int(lib().orc_double_to_bf16(float(d)))


def bf16_bits_to_float(h: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to float32 (bf16 is the top half of a binary32)."""
    return (np.asarray(h, np.uint16).astype(np.uint32) << 16).view(np.float32)
