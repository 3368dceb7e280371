"""bsm_softmax_noalloc: the entry point for callers that cannot allocate
device memory (code inside a pre-reserved pool or arena, or a path that
must not add the device-wide synchronisation of cudaMalloc/cudaFree).  Its
scratch is a fixed array inside the library instead of a plan's table.

It runs the planned dynamic schedule's kernel, row routine and patches, so
its output must equal bsm_softmax_ex(POLICY_DYNAMIC)'s bit for bit, and the
oracle's within the usual tolerance.

This file is collected last on purpose, so that a run stopping at the first
failure has run every other test first; the GPU test passes both alone in a
fresh process and after the rest of the suite."""
import ctypes

import pytest

from paper_2002_07062_gb300 import bsm, workload


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()


def test_oversized_batch_is_rejected_before_any_device_work():
    # 65537 patches of 32 fp32 rows of 512 elements (one 64 KiB stage each):
    # one more than the scratch holds
    rows = 32 * (bsm.NOALLOC_MAX_PATCHES + 1)
    rc = bsm.lib().bsm_softmax_noalloc(ctypes.c_void_p(256), ctypes.c_void_p(1 << 40), 1, rows,
                                       512, bsm.F32, 0, None)
    assert rc == bsm.ERR_TOO_LARGE
    assert "scratch" in bsm.status_string(rc)
    assert bsm.lib().bsm_softmax_noalloc(None, None, 0, 4, 4, bsm.F32, 0, None) == bsm.OK
    assert bsm.lib().bsm_softmax_noalloc(0, 0, 1, 4, 4, 3, 0, None) == bsm.ERR_INVALID_ARG


@pytest.mark.parametrize("dtype,es", [(bsm.F32, 4), (bsm.BF16, 2)])
def test_row_past_the_stage_limit_is_rejected_before_any_device_work(dtype, es):
    # the longest row that fits one stage passes these host checks (on a
    # machine without a GPU it then fails at the device query); one vector
    # more is refused as unsupported before the device is touched
    C = bsm.NOALLOC_MAX_ROW_BYTES // es
    rc = bsm.lib().bsm_softmax_noalloc(ctypes.c_void_p(256), ctypes.c_void_p(1 << 40), 1, 2,
                                       C + 16 // es, dtype, 0, None)
    assert rc == bsm.ERR_UNSUPPORTED
    # a huge batch of over-long rows: the row limit answers first, and nothing
    # multiplies rows by the row length on the way
    rc = bsm.lib().bsm_softmax_noalloc(ctypes.c_void_p(256), ctypes.c_void_p(1 << 40), 1 << 30,
                                       1 << 30, (1 << 31) - 16, dtype, 0, None)
    assert rc == bsm.ERR_UNSUPPORTED


def _cases():
    return [workload.uniform("noalloc fp32", workload.F32, 24, 96, 512, 3.0, 0xA11C0),
            workload.uniform("noalloc bf16 causal", workload.BF16, 7, 70, 384, 8.0, 0xA11C1,
                             workload.CAUSAL),
            # small batch: patches capped so that every SM gets one
            workload.uniform("noalloc fp32 8 x 64x64", workload.F32, 8, 64, 64, 1.0, 0xA11C2),
            # the longest row of one stage (113 KiB), fp32 shared-memory routine
            workload.uniform("noalloc fp32 longest row", workload.F32, 3, 5,
                             bsm.NOALLOC_MAX_ROW_BYTES // 4, 2.0, 0xA11C3),
            # many tiny bf16 slices, patches spanning slices
            workload.uniform("noalloc bf16 4096 x 32x128", workload.BF16, 4096, 32, 128, 1.0,
                             0xA11C4)]


@pytest.mark.gpu
def test_noalloc_matches_the_planned_entry_point_twice():
    import torch
    from gpu_util import bits, check_all_against_oracle, to_device, to_host
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()
    for w in _cases():
        w.materialize()
        x = to_device(w.x)
        R, C = int(w.rows[0]), int(w.cols[0])
        ref = torch.full_like(x, float("nan"))
        bsm.bsm_softmax_ex(x, ref, w.nslices, R, C, w.dtype, bsm.POLICY_DYNAMIC, w.flags)
        for call in range(2):            # two calls in a row share the scratch
            y = torch.full_like(x, float("nan"))
            rc = bsm.lib().bsm_softmax_noalloc(x.data_ptr(), y.data_ptr(), w.nslices, R, C,
                                               w.dtype, w.flags, None)
            assert rc == bsm.OK, bsm.status_string(rc)
            torch.cuda.synchronize()
            # the same kernel, routine and patches as the planned dynamic path
            assert torch.equal(bits(y), bits(ref)), (w.name, call)
            check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


@pytest.mark.gpu
def test_noalloc_timeout_is_reported_sticky_and_cleared():
    """A wait that runs out inside bsm_softmax_noalloc's kernel (a stage the
    test hook never fills; nothing faults) reaches bsm_device_status, stays
    there across later good calls, and bsm_device_status_clear removes it."""
    import time
    import torch
    from gpu_util import check_all_against_oracle, to_device, to_host
    torch.cuda.set_device(0)
    w = workload.uniform("noalloc status", workload.F32, 6, 64, 512, 2.0, 0xA11C5).materialize()
    x = to_device(w.x)
    y = torch.zeros_like(x)
    bsm.bsm_device_status_clear()
    bsm.bsm_plan_debug(None, bsm.DEBUG_WITHHOLD_STAGE, 100_000_000)     # 0.1 s waits
    try:
        t0 = time.time()
        rc = bsm.lib().bsm_softmax_noalloc(x.data_ptr(), y.data_ptr(), 6, 64, 512, bsm.F32, 0,
                                           None)
        assert rc == bsm.OK
        torch.cuda.synchronize()
        assert time.time() - t0 < 5.0
    finally:
        bsm.bsm_plan_debug(None, bsm.DEBUG_NONE)
    assert bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    # a good call afterwards computes the right result; the bit stays
    y.fill_(float("nan"))
    assert bsm.lib().bsm_softmax_noalloc(x.data_ptr(), y.data_ptr(), 6, 64, 512, bsm.F32, 0,
                                         None) == bsm.OK
    torch.cuda.synchronize()
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    bsm.bsm_device_status_clear()
    assert bsm.bsm_device_status() == 0
