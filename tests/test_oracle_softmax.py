"""Pins of the double-precision softmax oracle against things other than itself.

The paper names SOFTMAX on every 512 x 512 slice (Sec. 2; Sec. 6 table) but
prints no formula and no numbers, so the oracle is pinned to:
  * brute force: exp(v_c) / sum exp(v_c') evaluated with 50-digit decimals,
    WITHOUT the max shift, on tiny slices (catches a wrong axis, a dropped
    term, a wrong mask direction or row index, a transposed operand);
  * closed forms and special cases with exact answers;
  * invariants (rows sum to 1, per-row shift invariance);
  * a library routine for the bf16 rounding (torch's float32 -> bfloat16).
"""
import math
from decimal import Decimal, getcontext

import numpy as np
import pytest

from oracle import softmax as O

getcontext().prec = 50


def _dec_softmax_row(vals, row_in_slice=0, causal=False):
    """Definition of softmax along one row, in 50-digit decimal, no shift."""
    ex = []
    for c, v in enumerate(vals):
        if causal and c > row_in_slice:
            ex.append(Decimal(0))
        else:
            ex.append(Decimal(float(v)).exp())
    s = sum(ex)
    return [e / s for e in ex]


def _bf16_vals(bits):
    return O.bf16_bits_to_float(bits).astype(np.float64)


def _random_tiny(rng, shapes, dtype):
    rows = np.array([r for r, _ in shapes], np.int32)
    cols = np.array([c for _, c in shapes], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)
    vals = rng.normal(0.0, 3.0, int(sizes.sum())).astype(np.float32)
    if dtype == O.BF16:
        bits = (vals.view(np.uint32) >> 16).astype(np.uint16)
        return bits, off, rows, cols
    return vals, off, rows, cols


@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
@pytest.mark.parametrize("causal", [False, True])
def test_bruteforce_decimal_ragged_tiny(dtype, causal):
    rng = np.random.default_rng(7 + dtype + 2 * causal)
    shapes = [(3, 5), (8, 8), (1, 7), (6, 2), (4, 8), (5, 3)]
    x, off, rows, cols = _random_tiny(rng, shapes, dtype)
    y64, yout = O.softmax_batched(x, off, rows, cols, flags=O.CAUSAL if causal else 0)
    xv = _bf16_vals(x) if dtype == O.BF16 else x.astype(np.float64)
    for s, (R, C) in enumerate(shapes):
        for r in range(R):
            base = int(off[s]) + r * C
            ref = _dec_softmax_row(xv[base:base + C], r, causal)
            for c in range(C):
                got = y64[base + c]
                if causal and c > r:
                    assert got == 0.0
                    continue
                exact = ref[c]
                assert abs(Decimal(got) - exact) <= Decimal("4e-15") * exact, (s, r, c)


def test_bruteforce_decimal_workload1_full():
    """Every element of the 8 x 64x64 fp32 workload against the decimal definition."""
    from paper_2002_07062_gb300 import workload as W
    w = W.config(1).materialize()
    y64, yout = O.softmax_batched(w.x, w.offsets, w.rows, w.cols)
    x = w.x.astype(np.float64).reshape(-1, 64)
    y = y64.reshape(-1, 64)
    worst = 0.0
    for r in range(0, x.shape[0], 3):   # every third row keeps this a second or so
        ref = _dec_softmax_row(x[r])
        for c in range(64):
            rel = abs(Decimal(y[r, c]) - ref[c]) / ref[c]
            worst = max(worst, float(rel))
    assert worst <= 4e-15
    # the rounded output is the double result rounded to nearest fp32
    assert np.array_equal(yout, y64.astype(np.float32))


def test_rows_sum_to_one_and_thread_count_independent():
    rng = np.random.default_rng(3)
    x = rng.normal(0, 8, 37 * 300).astype(np.float32)
    rows, cols, off = [37], [300], [0]
    a, _ = O.softmax_batched(x, off, rows, cols, nthreads=1)
    b, _ = O.softmax_batched(x, off, rows, cols, nthreads=7)
    assert np.array_equal(a, b)
    s = a.reshape(37, 300).sum(axis=1)
    assert np.max(np.abs(s - 1.0)) <= 1e-12


def test_shift_invariance_is_exact():
    """x + k_r per row (k_r exact in fp32) gives bit-identical double results."""
    rng = np.random.default_rng(11)
    R, C = 16, 96
    x = (rng.integers(-4096, 4096, R * C) / 512.0).astype(np.float32)   # exact grid
    k = rng.integers(-32, 32, R).astype(np.float32)
    xs = (x.reshape(R, C) + k[:, None]).reshape(-1).astype(np.float32)
    assert np.array_equal(xs.astype(np.float64).reshape(R, C) - k[:, None],
                          x.astype(np.float64).reshape(R, C))           # shift exact
    a, _ = O.softmax_batched(x, [0], [R], [C])
    b, _ = O.softmax_batched(xs, [0], [R], [C])
    assert np.array_equal(a, b)


@pytest.mark.parametrize("C", [1, 2, 64, 512, 4096])
@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_constant_row_gives_exactly_one_over_C(C, dtype):
    x = np.full(C, 1.75, np.float32)
    if dtype == O.BF16:
        x = (x.view(np.uint32) >> 16).astype(np.uint16)
    y64, yout = O.softmax_row(x)
    assert np.all(y64 == 1.0 / C)
    if dtype == O.F32:
        assert np.all(yout == np.float32(1.0 / C))
    else:
        assert np.all(O.bf16_bits_to_float(yout) == np.float32(1.0 / C))


def test_one_hot_and_two_way_split_are_exact():
    x = np.full(33, -np.inf, np.float32)
    x[17] = 5.0
    y64, _ = O.softmax_row(x)
    assert y64[17] == 1.0 and np.all(np.delete(y64, 17) == 0.0)
    x[4] = 5.0
    y64, _ = O.softmax_row(x)
    assert y64[4] == 0.5 and y64[17] == 0.5 and np.count_nonzero(y64) == 2


def test_closed_form_log_ratios():
    """v = [0, ln 2, ln 3] gives y proportional to 1 : 2 : 3."""
    x = np.array([0.0, math.log(2.0), math.log(3.0)], np.float32)
    y64, _ = O.softmax_row(x)
    assert np.allclose(y64, [1 / 6, 2 / 6, 3 / 6], rtol=2e-7, atol=0)


def test_causal_row_zero_is_one_hot_in_every_slice():
    rng = np.random.default_rng(5)
    B, R, C = 3, 5, 9
    x = rng.normal(0, 8, B * R * C).astype(np.float32)
    y64, _ = O.softmax_batched(x, np.arange(B) * R * C, [R] * B, [C] * B, flags=O.CAUSAL)
    y = y64.reshape(B, R, C)
    assert np.all(y[:, 0, 0] == 1.0) and np.all(y[:, 0, 1:] == 0.0)
    # row r keeps columns 0..r; the rest are exactly zero
    for r in range(R):
        assert np.all(y[:, r, r + 1:] == 0.0)
        assert np.all(y[:, r, :r + 1] > 0.0)


def test_non_finite_rows_follow_the_formula():
    nan_row = np.array([0.0, np.nan, 1.0], np.float32)
    assert np.all(np.isnan(O.softmax_row(nan_row)[0]))
    inf_row = np.array([0.0, np.inf, 1.0], np.float32)
    assert np.all(np.isnan(O.softmax_row(inf_row)[0]))
    all_masked = np.full(4, -np.inf, np.float32)
    assert np.all(np.isnan(O.softmax_row(all_masked)[0]))
    # a NaN at a causally masked position still poisons the row: v = x + (-inf)
    x = np.array([1.0, 2.0, np.nan], np.float32)
    assert np.all(np.isnan(O.softmax_row(x, row_in_slice=0, flags=O.CAUSAL)[0]))


def test_bf16_rounding_matches_torch_on_float32_values():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(19)
    bits = rng.integers(0, 2 ** 32, 20000, dtype=np.uint64).astype(np.uint32)
    f = bits.view(np.float32)
    f = f[np.isfinite(f)]
    specials = np.array([0.0, -0.0, 1.0, 1 + 2 ** -8, 1 + 3 * 2 ** -8, 2 ** -133, 2 ** -134,
                         3 * 2 ** -134, 2 ** -126, 3.3895e38, 1e-40, 0.1, 1 / 3],
                        np.float32)
    f = np.concatenate([f, specials])
    ref = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy()
    ref = ref.view(np.uint16)
    got = np.array([O.double_to_bf16(float(v)) for v in f], np.uint16)
    assert np.array_equal(got, ref)


def test_bf16_rounding_happens_once_from_double():
    # 1 + 2^-8 + 2^-40 lies above the halfway point between 1 and 1 + 2^-7;
    # rounding through float32 first would land exactly on the tie and go to 1.
    assert O.double_to_bf16(1 + 2 ** -8 + 2 ** -40) == 0x3F81
    assert O.double_to_bf16(1 + 2 ** -8) == 0x3F80          # tie -> even
    assert O.double_to_bf16(1 + 3 * 2 ** -8) == 0x3F82      # tie -> even
    assert O.double_to_bf16(2.0 ** -134) == 0x0000          # tie below min subnormal
    assert O.double_to_bf16(3 * 2.0 ** -134) == 0x0002
    assert O.double_to_bf16(float("inf")) == 0x7F80
    assert O.double_to_bf16(3.4e38) == 0x7F80               # past the largest finite


def test_bad_arguments_are_rejected():
    with pytest.raises(RuntimeError):
        O.softmax_batched(np.zeros(4, np.float32), [0], [2], [0])
