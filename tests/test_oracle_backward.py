"""Pins of the softmax backward oracle (vector-Jacobian product of the row
softmax; Sec. 1: the batch algorithms also run in the backward pass).

The main pin is independent of the formula the oracle uses: central finite
differences of the softmax DEFINITION, evaluated with 50-digit decimals,
give J^T dy directly; the oracle's dx from (y, dy) must match.  Exact
special cases with dyadic y fix the sign and every term."""
from decimal import Decimal, getcontext

import numpy as np
import pytest

from oracle import softmax as O

getcontext().prec = 50


def _dec_softmax(vals):
    ex = [Decimal(float(v)).exp() for v in vals]
    s = sum(ex)
    return [e / s for e in ex]


def _fd_vjp(x, dy, h=Decimal("1e-20")):
    """sum_k dy_k * d softmax_k / d x_c by central differences, in decimal."""
    out = []
    for c in range(len(x)):
        xp = [Decimal(float(v)) for v in x]
        xm = list(xp)
        xp[c] += h
        xm[c] -= h
        def sm(vs):
            ex = [v.exp() for v in vs]
            s = sum(ex)
            return [e / s for e in ex]
        yp, ym = sm(xp), sm(xm)
        out.append(sum(Decimal(float(dy[k])) * (yp[k] - ym[k]) for k in range(len(x))) / (2 * h))
    return out


@pytest.mark.parametrize("C", [1, 3, 8, 13])
def test_backward_matches_finite_differences_of_the_definition(C):
    rng = np.random.default_rng(100 + C)
    x = rng.normal(0, 2, C)
    dy = rng.normal(0, 1, C).astype(np.float32)
    y_exact = _dec_softmax(x)
    y32 = np.array([float(v) for v in y_exact], np.float32)
    d64, _ = O.softmax_backward_row(y32, dy)
    ref = _fd_vjp(x, dy)
    for c in range(C):
        # y was rounded to fp32 for the oracle: allow that rounding (~6e-8 relative)
        assert abs(d64[c] - float(ref[c])) <= 1e-6 * (1 + abs(float(ref[c]))), (C, c)


def test_exact_dyadic_cases():
    y = np.array([0.5, 0.25, 0.125, 0.125], np.float32)
    # constant upstream gradient: dx = 0 exactly (sum y = 1)
    d64, _ = O.softmax_backward_row(y, np.full(4, 3.0, np.float32))
    assert np.all(d64 == 0.0)
    # one-hot upstream gradient e_k: dx_c = y_c (delta_ck - y_k)
    for k in range(4):
        dy = np.zeros(4, np.float32)
        dy[k] = 1.0
        d64, _ = O.softmax_backward_row(y, dy)
        want = [float(y[c]) * ((1.0 if c == k else 0.0) - float(y[k])) for c in range(4)]
        assert list(d64) == want
    # the gradient sums to zero when sum(y) = 1 exactly
    dy = np.array([1.5, -2.0, 0.75, 4.0], np.float32)
    d64, _ = O.softmax_backward_row(y, dy)
    assert d64.sum() == 0.0


def test_batched_backward_equals_rows_and_rounds_once():
    rng = np.random.default_rng(7)
    shapes = [(3, 5), (4, 8), (1, 16)]
    sizes = [r * c for r, c in shapes]
    off = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    y = rng.random(sum(sizes)).astype(np.float32)
    dy = rng.normal(0, 1, sum(sizes)).astype(np.float32)
    d64, dout = O.softmax_backward_batched(y, dy, off, [r for r, _ in shapes],
                                           [c for _, c in shapes])
    for s, (R, C) in enumerate(shapes):
        for r in range(R):
            a = int(off[s]) + r * C
            yr, dyr = y[a:a + C].astype(np.float64), dy[a:a + C].astype(np.float64)
            dot = 0.0
            for c in range(C):
                dot += yr[c] * dyr[c]
            assert np.array_equal(d64[a:a + C], yr * (dyr - dot))
    assert np.array_equal(dout, d64.astype(np.float32))
    # bf16: rounding of the double result with the oracle's own RNE
    yb = (y.view(np.uint32) >> 16).astype(np.uint16)
    dyb = (dy.view(np.uint32) >> 16).astype(np.uint16)
    d64b, doutb = O.softmax_backward_batched(yb, dyb, off, [r for r, _ in shapes],
                                             [c for _, c in shapes])
    assert all(int(doutb[i]) == O.double_to_bf16(d64b[i]) for i in range(0, d64b.size, 7))
