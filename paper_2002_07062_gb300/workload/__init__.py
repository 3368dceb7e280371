"""Seeded synthetic workloads for the batched softmax (inputs only).

This module makes input numbers and slice shapes and nothing else: it holds
none of the softmax or scheduling arithmetic.  The CUDA path and the CPU
oracle both consume the host arrays it returns.

The five workloads follow the shapes of the paper's running example (Sec. 2:
384 slices of 512 x 512, softmax along the last dimension, as in BERT
attention scores) plus the small, bf16-causal, ragged and many-tiny-slices
variants used to exercise the scheduler.  Workload k draws its values with
seed 0x2002070600 + k.  No public dataset is involved: these synthetic arrays
stand in for attention scores.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass, field
from typing import Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_DIR = os.path.join(os.path.dirname(HERE), "_lib")
LIB = os.path.join(LIB_DIR, "libbsm_gen.so")
SRC = os.path.join(HERE, "gen.c")

F32 = 0
BF16 = 1
CAUSAL = 1
SEED_BASE = 0x2002070600

_lib = None


def build(force: bool = False) -> str:
    import subprocess
    os.makedirs(LIB_DIR, exist_ok=True)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= os.path.getmtime(SRC):
        return LIB
    tmp = LIB + ".tmp%d" % os.getpid()
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                    "-Wall", "-o", tmp, SRC, "-lm", "-lpthread"], check=True)
    os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    if _lib is None:
        path = LIB if os.path.exists(LIB) else build()
        L = ctypes.CDLL(path)
        L.gen_fill_normal.argtypes = [ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                      ctypes.c_uint64, ctypes.c_double, ctypes.c_double,
                                      ctypes.c_int64, ctypes.c_int]
        L.gen_fill_normal.restype = ctypes.c_int
        L.gen_ragged_shapes.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                        ctypes.c_uint64, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_int32, ctypes.c_int32]
        L.gen_ragged_shapes.restype = ctypes.c_int
        L.gen_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        L.gen_splitmix64.restype = ctypes.c_uint64
        L.gen_normal.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        L.gen_normal.restype = ctypes.c_double
        _lib = L
    return _lib


def fill_normal(n: int, dtype: int, seed: int, sigma: float = 1.0, mu: float = 0.0,
                index_base: int = 0, out: Optional[np.ndarray] = None,
                nthreads: Optional[int] = None) -> np.ndarray:
    """n draws of mu + sigma*N(0,1), as float32 or as bf16 bit patterns (uint16)."""
    np_dt = np.float32 if dtype == F32 else np.uint16
    if out is None:
        out = np.empty(n, np_dt)
    assert out.dtype == np_dt and out.size == n and out.flags.c_contiguous
    rc = lib().gen_fill_normal(out.ctypes.data, dtype, n, seed & ((1 << 64) - 1), mu, sigma,
                               index_base, nthreads or os.cpu_count() or 1)
    if rc:
        raise RuntimeError("gen_fill_normal failed: %d" % rc)
    return out


def ragged_shapes(nslices: int, seed: int, row_unit=64, row_steps=16, col_unit=64,
                  col_steps=32):
    rows = np.empty(nslices, np.int32)
    cols = np.empty(nslices, np.int32)
    rc = lib().gen_ragged_shapes(rows.ctypes.data, cols.ctypes.data, nslices,
                                 (seed ^ 0x5348415045) & ((1 << 64) - 1),
                                 row_unit, row_steps, col_unit, col_steps)
    if rc:
        raise RuntimeError("gen_ragged_shapes failed: %d" % rc)
    return rows, cols


@dataclass
class Workload:
    name: str
    dtype: int
    rows: np.ndarray      # int32 per slice
    cols: np.ndarray      # int32 per slice
    offsets: np.ndarray   # int64 element offset of each slice
    flags: int
    seed: int
    sigma: float
    x: Optional[np.ndarray] = field(default=None, repr=False)

    @property
    def nslices(self) -> int:
        return len(self.rows)

    @property
    def numel(self) -> int:
        if self.nslices == 0:
            return 0
        return int(self.offsets[-1] + int(self.rows[-1]) * int(self.cols[-1]))

    @property
    def esize(self) -> int:
        return 4 if self.dtype == F32 else 2

    @property
    def algorithmic_bytes(self) -> int:
        """Bytes one softmax pass must move: every input element read once and
        every output element written once."""
        return 2 * self.numel * self.esize

    @property
    def uniform(self) -> bool:
        return self.nslices > 0 and bool((self.rows == self.rows[0]).all()
                                         and (self.cols == self.cols[0]).all())

    def materialize(self, nthreads: Optional[int] = None) -> "Workload":
        if self.x is None:
            self.x = fill_normal(self.numel, self.dtype, self.seed, self.sigma,
                                 nthreads=nthreads)
        return self


def uniform(name: str, dtype: int, B: int, R: int, C: int, sigma: float, seed: int,
            flags: int = 0) -> Workload:
    rows = np.full(B, R, np.int32)
    cols = np.full(B, C, np.int32)
    offsets = np.arange(B, dtype=np.int64) * (R * C)
    return Workload(name, dtype, rows, cols, offsets, flags, seed, sigma)


def ragged(name: str, dtype: int, nslices: int, sigma: float, seed: int, flags: int = 0,
           row_steps: int = 16, col_steps: int = 32, row_unit: int = 64,
           col_unit: int = 64) -> Workload:
    rows, cols = ragged_shapes(nslices, seed, row_unit, row_steps, col_unit, col_steps)
    sizes = rows.astype(np.int64) * cols.astype(np.int64)
    offsets = np.zeros(nslices, np.int64)
    if nslices > 1:
        offsets[1:] = np.cumsum(sizes)[:-1]
    return Workload(name, dtype, rows, cols, offsets, flags, seed, sigma)


def config(k: int) -> Workload:
    """The five workloads (values are not generated until materialize())."""
    seed = SEED_BASE + k
    if k == 1:
        return uniform("fp32 8 x 64x64 N(0,1)", F32, 8, 64, 64, 1.0, seed)
    if k == 2:
        return uniform("fp32 384 x 512x512 3*N(0,1)", F32, 384, 512, 512, 3.0, seed)
    if k == 3:
        return uniform("bf16 384 x 512x512 N(0,8) causal", BF16, 384, 512, 512, 8.0, seed,
                       CAUSAL)
    if k == 4:
        return ragged("fp32 ragged 1000 slices R=64*U{1..16} C=64*U{1..32} N(0,2)", F32,
                      1000, 2.0, seed)
    if k == 5:
        return uniform("bf16 65536 x 32x128 N(0,1)", BF16, 65536, 32, 128, 1.0, seed)
    raise ValueError("workload %d does not exist (1..5)" % k)


def slice_sample(w: Workload, slices) -> Workload:
    """The same workload restricted to some of its slices, packed densely;
    the values are those of the full workload (same draw indices)."""
    slices = np.asarray(slices, np.int64)
    rows = w.rows[slices].copy()
    cols = w.cols[slices].copy()
    sizes = rows.astype(np.int64) * cols.astype(np.int64)
    offsets = np.zeros(len(slices), np.int64)
    if len(slices) > 1:
        offsets[1:] = np.cumsum(sizes)[:-1]
    np_dt = np.float32 if w.dtype == F32 else np.uint16
    x = np.empty(int(sizes.sum()), np_dt)
    for j, s in enumerate(slices):
        n = int(sizes[j])
        seg = x[offsets[j]:offsets[j] + n]
        if w.x is not None:
            seg[:] = w.x[w.offsets[s]:w.offsets[s] + n]
        else:
            fill_normal(n, w.dtype, w.seed, w.sigma, index_base=int(w.offsets[s]), out=seg)
    return Workload(w.name + " [sample of %d slices]" % len(slices), w.dtype, rows, cols,
                    offsets, w.flags, w.seed, w.sigma, x)


# ---------------------------------------------------------------------------
# Batched matrix product operands (Sec. 6 matrix-multiplication table).

@dataclass
class BmmWorkload:
    """B slices of A_s (M x K) and Bt_s (N x K), bf16, row-major, packed; the
    product is written as out_dtype (F32 or BF16).  kind "normal": N(0, sigma)
    draws; kind "int": the same draws rounded to integers in [-6, 6], so that
    every product and partial sum is exact in fp32."""
    name: str
    B: int
    M: int
    N: int
    K: int
    out_dtype: int
    seed: int
    sigma: float = 1.0
    kind: str = "normal"

    @property
    def flops(self) -> int:
        return 2 * self.B * self.M * self.N * self.K

    @property
    def algorithmic_bytes(self) -> int:
        """Both operands read once, the product written once."""
        out_es = 4 if self.out_dtype == F32 else 2
        return 2 * self.B * (self.M + self.N) * self.K + out_es * self.B * self.M * self.N

    def _draw(self, which: int, n: int, base: int, out=None) -> np.ndarray:
        seed = (self.seed * 2 + which) & ((1 << 64) - 1)
        if self.kind == "int":
            v = fill_normal(n, F32, seed, 2.0, index_base=base)
            v = np.clip(np.rint(v), -6, 6).astype(np.float32)
            bits16 = (v.view(np.uint32) >> 16).astype(np.uint16)
            if out is not None:
                out[:] = bits16
                return out
            return bits16
        return fill_normal(n, BF16, seed, self.sigma, index_base=base, out=out)

    def operands(self, slices=None):
        """(a_bits, bt_bits) as uint16 bf16 patterns, for all slices or for
        the listed ones (packed, same values as in the full tensors)."""
        mk, nk = self.M * self.K, self.N * self.K
        if slices is None:
            return self._draw(0, self.B * mk, 0), self._draw(1, self.B * nk, 0)
        slices = list(slices)
        a = np.empty(len(slices) * mk, np.uint16)
        bt = np.empty(len(slices) * nk, np.uint16)
        for j, s in enumerate(slices):
            self._draw(0, mk, s * mk, out=a[j * mk:(j + 1) * mk])
            self._draw(1, nk, s * nk, out=bt[j * nk:(j + 1) * nk])
        return a, bt


def bmm_config(k: int) -> BmmWorkload:
    """The paper's two batched products (Sec. 6), bf16 in, bf16 out."""
    if k == 1:
        return BmmWorkload("bf16 384 x (512x64)(64x512)", 384, 512, 512, 64, BF16, SEED_BASE + 101)
    if k == 2:
        return BmmWorkload("bf16 384 x (512x512)(512x64)", 384, 512, 64, 512, BF16, SEED_BASE + 102)
    raise ValueError("batched product %d does not exist (1..2)" % k)
