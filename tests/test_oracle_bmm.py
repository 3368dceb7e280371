"""Pins of the batched matrix-product oracle: a triple loop on tiny
operands, identity and permutation operands, and small-integer operands whose
products are exact."""
import numpy as np

from oracle import bmm_oracle as BO
from oracle import softmax as O


def _bits(x):
    x = np.asarray(x, np.float32)
    return (x.view(np.uint32) >> 16).astype(np.uint16)    # exact for bf16-representable values


def test_against_triple_loop():
    rng = np.random.default_rng(1)
    B, M, N, K = 2, 3, 4, 5
    a = O.bf16_bits_to_float(_bits(rng.normal(0, 1, (B, M, K)))).astype(np.float64)
    bt = O.bf16_bits_to_float(_bits(rng.normal(0, 1, (B, N, K)))).astype(np.float64)
    got = BO.bmm_f64(_bits(a), _bits(bt), B, M, N, K)
    ref = BO.bmm_naive(a, bt)
    assert np.allclose(got, ref, rtol=1e-15, atol=1e-15)


def test_identity_and_permutation():
    K = 8
    eye = np.eye(K)
    perm = np.eye(K)[[3, 1, 7, 0, 2, 6, 4, 5]]
    a = np.arange(1, 2 * K * K + 1, dtype=np.float64).reshape(2, K, K) / 8.0
    got = BO.bmm_f64(_bits(a), _bits(np.stack([eye, perm])), 2, K, K, K)
    assert np.array_equal(got[0], a[0])                     # A I^T = A
    assert np.array_equal(got[1], a[1] @ perm.T)            # columns permuted


def test_small_integers_are_exact_and_rounding():
    rng = np.random.default_rng(2)
    a = rng.integers(-8, 9, (1, 16, 64)).astype(np.float64)
    bt = rng.integers(-8, 9, (1, 32, 64)).astype(np.float64)
    got = BO.bmm_f64(_bits(a), _bits(bt), 1, 16, 32, 64)
    exact = np.einsum("smk,snk->smn", a, bt)
    assert np.array_equal(got, exact)
    r = BO.round_bf16(np.array([1.0, 257.0, 259.0, -3.0]))
    assert list(r) == [0x3F80, 0x4380, 0x4382, 0xC040]     # 257 -> 256 (tie, even), 259 -> 260
