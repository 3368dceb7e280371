"""bmm_oracle.py -- TEST INFRASTRUCTURE ONLY.

The paper's second batch algorithm (Sec. 6, the matrix-multiplication table:
batch 384 of (512 x 64) x (64 x 512) and of (512 x 512) x (512 x 64)) is a
batched matrix product C_s = A_s B_s for every slice s.  The tensor-core
kernel reads both operands with the reduction dimension contiguous, so the
second operand is supplied as its transpose: for slice s, A_s is M x K
row-major, Bt_s is N x K row-major (B_s = Bt_s^T) and

    C_s[m, n] = sum_k A_s[m, k] * Bt_s[n, k]

evaluated here in double from exactly converted bf16 inputs (numpy's float64
matrix product is the summation step), then rounded once to the output type
(float32 by the C conversion, bf16 with the softmax oracle's own rounding).
Imported only by tests and bench.py's CPU leg.
"""
from __future__ import annotations

import numpy as np

from .softmax import bf16_bits_to_float, double_to_bf16


def bmm_f64(a_bits: np.ndarray, bt_bits: np.ndarray, B: int, M: int, N: int, K: int) -> np.ndarray:
    """a_bits: B*M*K bf16 bit patterns, bt_bits: B*N*K; returns B x M x N float64."""
    a = bf16_bits_to_float(a_bits).astype(np.float64).reshape(B, M, K)
    bt = bf16_bits_to_float(bt_bits).astype(np.float64).reshape(B, N, K)
    return np.matmul(a, np.transpose(bt, (0, 2, 1)))


def round_bf16(c: np.ndarray) -> np.ndarray:
    """Round every double to bf16 bits (the oracle's own round-to-nearest-even)."""
    flat = np.asarray(c, np.float64).reshape(-1)
    return np.array([double_to_bf16(float(v)) for v in flat], np.uint16).reshape(np.shape(c))


def bmm_naive(a: np.ndarray, bt: np.ndarray) -> np.ndarray:
    """Triple loop on tiny float64 inputs (B x M x K and B x N x K)."""
    B, M, K = a.shape
    N = bt.shape[1]
    c = np.zeros((B, M, N))
    for s in range(B):
        for m in range(M):
            for n in range(N):
                acc = 0.0
                for k in range(K):
                    acc += a[s, m, k] * bt[s, n, k]
                c[s, m, n] = acc
    return c
