"""GPU parity of the softmax backward pass (dx = y * (dy - <y, dy>) per row)
against the double-precision oracle, under every scheduling policy.

Tolerance, from the arithmetic of the kernel (fp32 products and sums, unit
roundoff u = 2^-24): the dot product goes through at most L roundings
(vector tree, per-lane sum, butterfly), the difference and the product one
each, so |dx - dx_exact| <= y * (L*u*sum|y*dy| + 2u(|dy| + |dot|)); checked
with a factor 2 margin.  bf16 outputs may in addition sit one bf16 unit in
the last place from the oracle's rounding."""
import numpy as np
import pytest

from gpu_util import bits, to_device, to_host
from oracle import softmax as O
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu

ALL = [bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR, bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF,
       bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX]
U = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()


def _inputs(w):
    """y = the oracle's forward output (in the io type), dy = N(0,1) draws."""
    _, y = O.softmax_batched(w.x, w.offsets, w.rows, w.cols, w.flags)
    dy = workload.fill_normal(w.numel, w.dtype, w.seed ^ 0xD1, 1.0)
    return y, dy


def _to_f64(a, dtype):
    return (O.bf16_bits_to_float(a) if dtype == workload.BF16 else a).astype(np.float64)


def _check(w, y, dy, dx_gpu, rows=None):
    d64, dround = O.softmax_backward_batched(y, dy, w.offsets, w.rows, w.cols)
    yf, df = _to_f64(y, w.dtype), _to_f64(dy, w.dtype)
    got = _to_f64(dx_gpu, w.dtype)
    worst = 0.0
    for s in range(w.nslices):
        R, C = int(w.rows[s]), int(w.cols[s])
        a = int(w.offsets[s])
        Y = yf[a:a + R * C].reshape(R, C)
        D = df[a:a + R * C].reshape(R, C)
        dot = (Y * D).sum(axis=1, keepdims=True)
        L = 3 + max(1, (C * (4 if w.dtype == workload.F32 else 2) // 16 + 31) // 32) + 5
        bound = 2 * Y * (L * U * np.abs(Y * D).sum(axis=1, keepdims=True)
                         + 2 * U * (np.abs(D) + np.abs(dot)))
        err = np.abs(got[a:a + R * C].reshape(R, C) - d64[a:a + R * C].reshape(R, C))
        if w.dtype == workload.BF16:
            ulp = np.abs(_to_f64(dround[a:a + R * C], w.dtype)).reshape(R, C) * 2.0 ** -7
            bound = bound + np.maximum(ulp, 2.0 ** -133)
        assert np.all(err <= bound), (s, float((err - bound).max()))
        worst = max(worst, float(err.max()))
    return worst


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
@pytest.mark.parametrize("col_steps", [160, 768])
def test_backward_ragged_every_routine(dtype, col_steps):
    import torch
    unit = 4 if dtype == workload.F32 else 8
    w = workload.ragged("bwd classes", dtype, 24, 2.0, 300 + col_steps + dtype, row_unit=1,
                        row_steps=60, col_unit=unit, col_steps=col_steps).materialize()
    y, dy = _inputs(w)
    yd, dyd = to_device(y), to_device(dy)
    outs = []
    for pol in ALL:
        dx = torch.full_like(yd, float("nan"))
        bsm.bsm_softmax_backward_ragged(yd, dyd, dx, w.offsets, w.rows, w.cols, w.dtype, pol)
        outs.append(dx)
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(bits(o), bits(outs[0]))
    _check(w, y, dy, to_host(outs[0]))
    assert bsm.bsm_device_status() == 0


@pytest.mark.parametrize("k", [2, 3])
def test_backward_full_size_uniform_and_in_place(k):
    import torch
    w = workload.config(k).materialize()
    R, C = int(w.rows[0]), int(w.cols[0])
    y, dy = _inputs(w)
    yd, dyd = to_device(y), to_device(dy)
    dx = torch.full_like(yd, float("nan"))
    bsm.bsm_softmax_backward(yd, dyd, dx, w.nslices, R, C, w.dtype, bsm.POLICY_DYNAMIC)
    torch.cuda.synchronize()
    assert not torch.isnan(dx).any()
    # a sample of slices against the oracle, all rows of each
    pick = list(range(0, w.nslices, 29))
    sw = workload.slice_sample(w, pick)
    ys = np.concatenate([y[w.offsets[s]:w.offsets[s] + R * C] for s in pick])
    dys = np.concatenate([dy[w.offsets[s]:w.offsets[s] + R * C] for s in pick])
    dxh = to_host(dx)
    dxs = np.concatenate([dxh[w.offsets[s]:w.offsets[s] + R * C] for s in pick])
    _check(sw, ys, dys, dxs)
    # in place into dy gives the same bits
    bsm.bsm_softmax_backward(yd, dyd, dyd, w.nslices, R, C, w.dtype, bsm.POLICY_RR)
    torch.cuda.synchronize()
    assert torch.equal(bits(dyd), bits(dx))
    assert bsm.bsm_device_status() == 0


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
def test_backward_rows_longer_than_half_a_stage(dtype):
    """Rows whose y and dy do not fit one stage are streamed twice in chunks
    (the dot product, then dx); same tolerance, all policies bit-identical,
    and in place into dy."""
    import torch
    es = 4 if dtype == workload.F32 else 2
    half = bsm.bsm_max_row_bytes() // 2 // es          # elements in half a stage
    for B, R, C in [(2, 3, half + 16 // es), (1, 2, 262144), (3, 1, 100000 // 8 * 8)]:
        w = workload.uniform("bwd long", dtype, B, R, C, 3.0, 0xB10 + C).materialize()
        y, dy = _inputs(w)
        yd, dyd = to_device(y), to_device(dy)
        p = bsm.bsm_plan_create(yd, torch.empty_like(yd), w.rows, w.cols, dtype,
                                bsm.POLICY_DYNAMIC, op=bsm.OP_BACKWARD, x2=dyd)
        assert p.stats()["long_items"] == B * R
        p.close()
        outs = []
        for pol in ALL:
            dx = torch.full_like(yd, float("nan"))
            bsm.bsm_softmax_backward(yd, dyd, dx, B, R, C, dtype, pol)
            outs.append(dx)
        torch.cuda.synchronize()
        for o in outs[1:]:
            assert torch.equal(bits(o), bits(outs[0]))
        _check(w, y, dy, to_host(outs[0]))
        dyd2 = dyd.clone()
        bsm.bsm_softmax_backward(yd, dyd2, dyd2, B, R, C, dtype, bsm.POLICY_DYNAMIC)
        torch.cuda.synchronize()
        assert torch.equal(bits(dyd2), bits(outs[0]))
    assert bsm.bsm_device_status() == 0


def test_backward_mixed_short_and_long_rows():
    import torch
    rows = np.array([4, 1, 3, 2, 5, 1], np.int32)
    cols = np.array([64, 200000, 2048, 30000, 512, 16], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)
    w = workload.Workload("bwd mixed long", workload.F32, rows, cols, off, 0, 0x4D18, 2.0)
    w.materialize()
    y, dy = _inputs(w)
    yd, dyd = to_device(y), to_device(dy)
    outs = []
    for pol in ALL:
        dx = torch.full_like(yd, float("nan"))
        bsm.bsm_softmax_backward_ragged(yd, dyd, dx, w.offsets, w.rows, w.cols, w.dtype, pol)
        outs.append(dx)
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(bits(o), bits(outs[0]))
    _check(w, y, dy, to_host(outs[0]))
    assert bsm.bsm_device_status() == 0


@pytest.mark.parametrize("chunks", [2, 3])
def test_backward_many_long_rows_one_launch(chunks):
    """Two waves of backward long rows: each row streams twice in one launch,
    the second pass from its last chunk (still staged) backwards."""
    import torch
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    half = bsm.bsm_max_row_bytes() // 2 // 4
    R, C = 2 * n_sm + 8, (chunks - 1) * half + 4
    w = workload.uniform("bwd many long", workload.F32, 1, R, C, 3.0, 0xB77 + chunks).materialize()
    y, dy = _inputs(w)
    yd, dyd = to_device(y), to_device(dy)
    outs = []
    for pol in ALL:
        dx = torch.full_like(yd, float("nan"))
        bsm.bsm_softmax_backward(yd, dyd, dx, 1, R, C, workload.F32, pol)
        outs.append(dx)
    torch.cuda.synchronize()
    for o in outs[1:]:
        assert torch.equal(bits(o), bits(outs[0]))
    _check(w, y, dy, to_host(outs[0]))
    assert bsm.bsm_device_status() == 0
