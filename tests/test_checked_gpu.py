"""The self-checking kernel instances (bsm_set_device_checks): every shared
memory read, global store and bulk copy is checked against the stage and
buffer extents before it happens.  Run over workloads that reach every row
routine, the causal classes, long rows in both modes and the backward pass,
they must record no violation and give the same bits as the unchecked
kernels."""
import numpy as np
import pytest

from gpu_util import bits, run, to_device
from oracle import softmax as O
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def checks_off_afterwards():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()
    yield
    bsm.bsm_set_device_checks(False)


def _both(fn):
    """fn() run unchecked, then checked; returns the two outputs."""
    import torch
    bsm.bsm_set_device_checks(False)
    a = fn()
    bsm.bsm_set_device_checks(True)
    b = fn()
    torch.cuda.synchronize()
    bsm.bsm_set_device_checks(False)
    assert bsm.bsm_device_status() == 0, bsm.bsm_device_debug()
    return a, b


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
@pytest.mark.parametrize("flags", [0, workload.CAUSAL])
@pytest.mark.parametrize("col_steps", [160, 768])
def test_checked_forward_every_routine(dtype, flags, col_steps):
    unit = 4 if dtype == workload.F32 else 8
    w = workload.ragged("checked", dtype, 24, 2.0, 900 + col_steps + dtype + flags, flags,
                        row_unit=1, row_steps=60, col_unit=unit, col_steps=col_steps).materialize()
    x = to_device(w.x)
    for pol in (bsm.POLICY_DYNAMIC, bsm.POLICY_RR, bsm.POLICY_CBMF_LB):
        a, b = _both(lambda: run(w, x, pol))
        assert __import__("torch").equal(bits(a), bits(b))


@pytest.mark.parametrize("R,caps", [(3, 1), (400, 1), (400, 2)])
def test_checked_long_rows(R, caps):
    """3 rows: segments over two launches; 400 rows: one launch per row, of
    two chunks (staged whole between the passes) or three (the last chunk
    kept, the others copied again)."""
    import torch
    es = 4
    C = caps * (bsm.bsm_max_row_bytes() // es) + 64
    w = workload.uniform("checked long", workload.F32, 1, R, C, 2.0, 0xC4E + R).materialize()
    x = to_device(w.x)
    a, b = _both(lambda: run(w, x, bsm.POLICY_DYNAMIC))
    assert torch.equal(bits(a), bits(b))


def test_checked_backward_short_and_long():
    import torch
    rows = np.array([3, 1, 2, 5], np.int32)
    cols = np.array([512, 40000, 2048, 96], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)
    w = workload.Workload("checked bwd", workload.F32, rows, cols, off, 0, 0xC4F, 2.0)
    w.materialize()
    _, y = O.softmax_batched(w.x, w.offsets, w.rows, w.cols, w.flags)
    dy = workload.fill_normal(w.numel, w.dtype, 0xC50, 1.0)
    yd, dyd = to_device(y), to_device(dy)

    def bwd():
        dx = torch.full_like(yd, float("nan"))
        bsm.bsm_softmax_backward_ragged(yd, dyd, dx, w.offsets, w.rows, w.cols, w.dtype,
                                        bsm.POLICY_DYNAMIC)
        return dx
    a, b = _both(bwd)
    assert torch.equal(bits(a), bits(b))


def test_checked_group_rows():
    """Rows split over groups of CTAs (19 of the 25 groups of 6 on 152 SMs): the
    self-checking group kernel checks its bulk copies, stage reads and
    stores, and gives the same bits."""
    import torch
    w = workload.uniform("checked group", workload.F32, 1, 19, 98304, 2.0, 0xC51).materialize()
    x = to_device(w.x)
    a, b = _both(lambda: run(w, x, bsm.POLICY_DYNAMIC))
    assert torch.equal(bits(a), bits(b))
