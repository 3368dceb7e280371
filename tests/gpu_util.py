"""Helpers shared by the GPU parity tests: move workloads to the device, run
the C ABI under a policy, and compare sampled or full outputs with the
double-precision oracle."""
from __future__ import annotations

import numpy as np

from oracle import softmax as O
from paper_2002_07062_gb300 import bsm, workload

FP32_TOL = 2e-6      # max |y_gpu - y_oracle| for fp32 output
BF16_ULPS = 1        # max distance in bf16 units in the last place


def to_device(a: np.ndarray):
    import torch
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).cuda().view(torch.bfloat16)
    return torch.from_numpy(a).cuda()


def to_host(t) -> np.ndarray:
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def bits(t):
    import torch
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


def is_packed(w: workload.Workload) -> bool:
    if w.nslices == 0:
        return True
    sizes = w.rows.astype(np.int64) * w.cols.astype(np.int64)
    expect = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    return bool(np.array_equal(expect, w.offsets))


def run(w: workload.Workload, x, policy: int, y=None, stream=None, force_ragged=False):
    """Softmax of workload w (device input x) under `policy`; returns y."""
    import torch
    if y is None:
        y = torch.full_like(x, float("nan"))
    if w.uniform and is_packed(w) and not force_ragged:
        bsm.bsm_softmax_ex(x, y, w.nslices, int(w.rows[0]), int(w.cols[0]), w.dtype, policy,
                           w.flags, stream)
    else:
        bsm.bsm_softmax_ragged(x, y, w.offsets, w.rows, w.cols, w.dtype, policy, w.flags, stream)
    return y


def row_starts(w: workload.Workload):
    """(global row id -> slice, row in slice) helpers: cumulative row counts."""
    return np.concatenate([[0], np.cumsum(w.rows.astype(np.int64))])


def sample_rows(w: workload.Workload, n: int, seed: int):
    """n (slice, row) pairs: the first and last row of some slices plus random rows."""
    rng = np.random.default_rng(seed)
    base = row_starts(w)
    total = int(base[-1])
    picks = set()
    for s in rng.choice(w.nslices, size=min(w.nslices, n // 4 + 1), replace=False):
        if w.rows[s] > 0:
            picks.add((int(s), 0))
            picks.add((int(s), int(w.rows[s]) - 1))
    while len(picks) < n and total > 0:
        g = int(rng.integers(0, total))
        s = int(np.searchsorted(base, g, side="right") - 1)
        picks.add((s, g - int(base[s])))
    return sorted(picks)


def check_rows_against_oracle(w: workload.Workload, y_host: np.ndarray, pairs):
    """Compare the rows `pairs` of y_host with the oracle; returns the worst
    error (fp32: absolute; bf16: ulps)."""
    worst = 0.0
    for s, r in pairs:
        C = int(w.cols[s])
        a = int(w.offsets[s]) + r * C
        y64, yr = O.softmax_row(w.x[a:a + C], r, w.flags)
        got = y_host[a:a + C]
        if w.dtype == workload.F32:
            d = np.abs(got.astype(np.float64) - y64)
            nanmask = np.isnan(y64)
            assert np.array_equal(np.isnan(got), nanmask), (s, r)
            e = float(np.max(d[~nanmask])) if (~nanmask).any() else 0.0
            assert e <= FP32_TOL, (s, r, e)
        else:
            gi = got.astype(np.int32)
            wi = yr.astype(np.int32)
            nan_g = (gi & 0x7F80) == 0x7F80
            nan_w = (wi & 0x7F80) == 0x7F80
            assert np.array_equal(nan_g & ((gi & 0x7F) != 0), nan_w & ((wi & 0x7F) != 0)), (s, r)
            ok = ~(nan_w & ((wi & 0x7F) != 0))
            e = float(np.max(np.abs(gi[ok] - wi[ok]))) if ok.any() else 0.0
            assert e <= BF16_ULPS, (s, r, e)
        worst = max(worst, e)
    return worst


def check_all_against_oracle(w: workload.Workload, y_host: np.ndarray):
    y64, yr = O.softmax_batched(w.x, w.offsets, w.rows, w.cols, w.flags)
    if is_packed(w) and w.numel == w.x.size:
        covered = slice(None)                  # the slices cover the whole array
    else:
        covered = np.zeros(w.x.size, bool)
        for s in range(w.nslices):
            n = int(w.rows[s]) * int(w.cols[s])
            covered[int(w.offsets[s]):int(w.offsets[s]) + n] = True
    if w.dtype == workload.F32:
        g = y_host[covered].astype(np.float64)
        o = y64[covered]
        nan_o = np.isnan(o)
        if nan_o.any():
            assert np.array_equal(np.isnan(g), nan_o)
            m = ~nan_o
            err = float(np.max(np.abs(g[m] - o[m]))) if m.any() else 0.0
        else:
            # no NaN expected: a NaN in g makes the maximum NaN, which fails
            np.subtract(g, o, out=g)
            np.abs(g, out=g)
            err = float(np.max(g)) if g.size else 0.0
        assert err <= FP32_TOL, err
        return err
    gi = y_host[covered].astype(np.int32)
    wi = yr[covered].astype(np.int32)
    np.subtract(gi, wi, out=gi)
    np.abs(gi, out=gi)
    err = float(np.max(gi)) if gi.size else 0.0
    assert err <= BF16_ULPS, err
    return err


def check_every_element_against_oracle(w: workload.Workload, y_host: np.ndarray,
                                       max_elems: int = 1 << 26):
    """check_all_against_oracle over every slice of w, in groups of slices of
    at most about max_elems elements (the oracle's double-precision output of
    a whole 4.6 GB workload would need tens of GB of host memory at once).
    Returns the worst error (fp32: absolute; bf16: ulps)."""
    worst = 0.0
    packed = is_packed(w)

    def n_last(s):
        return int(w.rows[s]) * int(w.cols[s])
    s0 = 0
    while s0 < w.nslices:
        s1, n = s0, 0
        while s1 < w.nslices and (s1 == s0 or n + int(w.rows[s1]) * int(w.cols[s1]) <= max_elems):
            n += int(w.rows[s1]) * int(w.cols[s1])
            s1 += 1
        if packed:
            # consecutive slices are one contiguous range of x and y
            a, b = int(w.offsets[s0]), int(w.offsets[s1 - 1]) + n_last(s1 - 1)
            sub = workload.Workload(w.name, w.dtype, w.rows[s0:s1], w.cols[s0:s1],
                                    w.offsets[s0:s1] - a, w.flags, w.seed, w.sigma, w.x[a:b])
            ys = y_host[a:b]
        else:
            idx = np.arange(s0, s1)
            sub = workload.slice_sample(w, idx)
            ys = np.empty_like(sub.x)
            for j, s in enumerate(idx):
                m = n_last(s)
                ys[int(sub.offsets[j]):int(sub.offsets[j]) + m] = \
                    y_host[int(w.offsets[s]):int(w.offsets[s]) + m]
        worst = max(worst, check_all_against_oracle(sub, ys))
        s0 = s1
    return worst
