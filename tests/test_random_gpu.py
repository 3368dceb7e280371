"""Randomised parity: seeded random ragged batches -- dtype, causal flag,
policy, rows per slice, row length (now and then longer than a stage), gaps
between slices -- each compared element by element with the oracle and bit
for bit with the DYNAMIC policy; the backward pass the same way."""
import numpy as np
import pytest

from gpu_util import bits, check_all_against_oracle, run, to_device, to_host
from oracle import softmax as O
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu

POLICIES = [bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR, bsm.POLICY_CBMF, bsm.POLICY_CBMF_LB,
            bsm.POLICY_MINIMAX]


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()


def _random_batch(rng, dtype, flags):
    es = 4 if dtype == workload.F32 else 2
    unit = 16 // es
    long_c = bsm.bsm_max_row_bytes() // es + unit * int(rng.integers(1, 200))
    n = int(rng.integers(1, 40))
    rows = rng.integers(1, 300, n).astype(np.int32)
    cols = (unit * rng.integers(1, 512 // unit * 8 + 1, n)).astype(np.int32)
    if rng.random() < 0.3:                       # a few rows longer than a stage
        k = int(rng.integers(0, n))
        cols[k] = long_c
        rows[k] = int(rng.integers(1, 4))
    sizes = rows.astype(np.int64) * cols
    gaps = unit * rng.integers(0, 3, n)          # unused elements between slices
    off = np.zeros(n, np.int64)
    pos = 0
    for i in range(n):
        pos += int(gaps[i])
        off[i] = pos
        pos += int(sizes[i])
    w = workload.Workload("random", dtype, rows, cols, off, flags, int(rng.integers(1, 1 << 30)),
                          float(rng.choice([0.5, 2.0, 8.0])))
    w.x = workload.fill_normal(pos, dtype, w.seed, w.sigma)
    return w


@pytest.mark.parametrize("case", range(40))
def test_random_forward(case):
    import torch
    rng = np.random.default_rng(0xA11 + case)
    dtype = workload.F32 if case % 2 == 0 else workload.BF16
    flags = workload.CAUSAL if (case // 2) % 2 else 0
    w = _random_batch(rng, dtype, flags)
    x = to_device(w.x)
    ref = run(w, x, bsm.POLICY_DYNAMIC, force_ragged=True)
    pol = POLICIES[case % len(POLICIES)]
    y = run(w, x, pol, force_ragged=True)
    torch.cuda.synchronize()
    assert torch.equal(bits(y), bits(ref)), bsm.POLICY_NAMES[pol]
    check_all_against_oracle(w, to_host(ref))
    assert bsm.bsm_device_status() == 0


@pytest.mark.parametrize("case", range(12))
def test_random_backward(case):
    import torch
    rng = np.random.default_rng(0xB22 + case)
    dtype = workload.F32 if case % 2 == 0 else workload.BF16
    w = _random_batch(rng, dtype, 0)
    _, y = O.softmax_batched(w.x, w.offsets, w.rows, w.cols, 0)
    dy = workload.fill_normal(w.x.size, dtype, w.seed ^ 0x77, 1.0)
    yd, dyd = to_device(y), to_device(dy)
    outs = []
    for pol in (bsm.POLICY_DYNAMIC, POLICIES[case % len(POLICIES)]):
        dx = torch.zeros_like(yd)
        bsm.bsm_softmax_backward_ragged(yd, dyd, dx, w.offsets, w.rows, w.cols, dtype, pol)
        outs.append(dx)
    torch.cuda.synchronize()
    assert torch.equal(bits(outs[0]), bits(outs[1]))
    d64, _ = O.softmax_backward_batched(y, dy, w.offsets, w.rows, w.cols)
    got = to_host(outs[0])
    got = (O.bf16_bits_to_float(got) if dtype == workload.BF16 else got).astype(np.float64)
    yf = (O.bf16_bits_to_float(y) if dtype == workload.BF16 else y).astype(np.float64)
    df = (O.bf16_bits_to_float(dy) if dtype == workload.BF16 else dy).astype(np.float64)
    for s in range(w.nslices):
        R, C, a = int(w.rows[s]), int(w.cols[s]), int(w.offsets[s])
        Y = yf[a:a + R * C].reshape(R, C)
        D = df[a:a + R * C].reshape(R, C)
        dot = (Y * D).sum(axis=1, keepdims=True)
        L = 3 + max(1, (C * (4 if dtype == workload.F32 else 2) // 16 + 31) // 32) + 5 + 16
        bound = 2 * Y * (L * 2.0 ** -24 * np.abs(Y * D).sum(axis=1, keepdims=True)
                         + 2 * 2.0 ** -24 * (np.abs(D) + np.abs(dot)))
        if dtype == workload.BF16:
            bound = bound + np.maximum(np.abs(d64[a:a + R * C].reshape(R, C)) * 2.0 ** -7, 2.0 ** -133)
        err = np.abs(got[a:a + R * C].reshape(R, C) - d64[a:a + R * C].reshape(R, C))
        assert np.all(err <= bound), (s, R, C, float((err - bound).max()))
    assert bsm.bsm_device_status() == 0
