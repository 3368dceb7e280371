"""Failure detection on the GPU without faulting it: a stage that is never
filled makes the bounded pipeline waits run out (BSM_DEV_TIMEOUT), and a
patch entry pointing past the buffers is skipped by the kernel's bounds check
(BSM_DEV_BOUNDS).  In both cases the context stays usable: a normal launch
right after gives correct results."""
import numpy as np
import pytest

from gpu_util import check_all_against_oracle, to_device, to_host
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    yield
    bsm.bsm_device_status_clear()


def _w():
    return workload.uniform("fail", workload.F32, 6, 64, 512, 2.0, 0xFA11).materialize()


def test_withheld_stage_times_out_and_context_survives():
    import time
    import torch
    w = _w()
    x = to_device(w.x)
    y = torch.zeros_like(x)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_DYNAMIC)
    bsm.bsm_plan_debug(p, bsm.DEBUG_WITHHOLD_STAGE, 100_000_000)      # 0.1 s waits
    t0 = time.time()
    p.execute()
    torch.cuda.synchronize()
    assert time.time() - t0 < 5.0
    st = bsm.bsm_device_status()
    assert st & bsm.DEV_TIMEOUT
    bsm.bsm_plan_debug(p, bsm.DEBUG_NONE)
    bsm.bsm_device_status_clear()
    y.fill_(float("nan"))
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y))
    p.close()


def test_corrupted_patch_is_skipped_with_bounds_status():
    import torch
    w = _w()
    x = to_device(w.x)
    sentinel = -7.0
    y = torch.full_like(x, sentinel)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_RR)
    n = p.stats()["n_items"]
    bsm.bsm_plan_debug(p, bsm.DEBUG_CORRUPT_PATCH, n // 2)
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() & bsm.DEV_BOUNDS
    yh = to_host(y).reshape(-1, 512)
    untouched = np.all(yh == sentinel, axis=1)
    rows_per_patch = (w.rows[0] * w.nslices) // n
    assert untouched.sum() == rows_per_patch                  # exactly one patch skipped
    # every other row is right
    ok = ~untouched
    from oracle import softmax as O
    y64, _ = O.softmax_batched(w.x, w.offsets, w.rows, w.cols)
    err = np.max(np.abs(yh[ok].astype(np.float64) - y64.reshape(-1, 512)[ok]))
    assert err <= 2e-6
    p.close()
    bsm.bsm_device_status_clear()
    # a fresh plan on the same buffers is unaffected
    y2 = torch.full_like(x, float("nan"))
    bsm.bsm_softmax(x, y2, w.nslices, 64, 512, w.dtype, bsm.POLICY_DYNAMIC)
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y2))


def _w_long():
    """Two waves of rows just over a stage: the one-launch long-row path
    (rows staged whole between their passes)."""
    import torch
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    C = bsm.bsm_max_row_bytes() // 4 + 64
    return workload.uniform("fail long", workload.F32, 1, 2 * n_sm + 3, C, 2.0, 0xFA12).materialize()


def test_withheld_stage_times_out_on_long_rows():
    import time
    import torch
    w = _w_long()
    x = to_device(w.x)
    y = torch.zeros_like(x)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_DYNAMIC)
    assert p.stats()["long_items"] == int(w.rows[0]) and p.stats()["launches"] == 1
    bsm.bsm_plan_debug(p, bsm.DEBUG_WITHHOLD_STAGE, 100_000_000)      # 0.1 s waits
    t0 = time.time()
    p.execute()
    torch.cuda.synchronize()
    assert time.time() - t0 < 5.0
    assert bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    bsm.bsm_plan_debug(p, bsm.DEBUG_NONE)
    bsm.bsm_device_status_clear()
    y.fill_(float("nan"))
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y))
    p.close()


def test_corrupted_long_patch_is_skipped_with_bounds_status():
    import torch
    w = _w_long()
    C = int(w.cols[0])
    x = to_device(w.x)
    sentinel = -7.0
    y = torch.full_like(x, sentinel)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_RR)
    n = p.stats()["n_items"]
    assert n == int(w.rows[0])                                 # one patch per long row
    bsm.bsm_plan_debug(p, bsm.DEBUG_CORRUPT_PATCH, n // 2)
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() & bsm.DEV_BOUNDS
    yh = to_host(y).reshape(-1, C)
    untouched = np.all(yh == sentinel, axis=1)
    assert untouched.sum() == 1 and untouched[n // 2]
    from oracle import softmax as O
    y64, _ = O.softmax_batched(w.x, w.offsets, w.rows, w.cols)
    ok = ~untouched
    assert np.max(np.abs(yh[ok].astype(np.float64) - y64.reshape(-1, C)[ok])) <= 2e-6
    p.close()
    bsm.bsm_device_status_clear()


def test_whole_gpu_graph_and_debug_launches():
    """WHOLE_GPU plans run their per-slice launches as one captured graph; a
    plan under a debug setting launches kernel by kernel (the withheld stage
    times out), and back on the graph afterwards gives correct results."""
    import torch
    w = _w()
    x = to_device(w.x)
    y = torch.full_like(x, float("nan"))
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_WHOLE_GPU)
    assert p.stats()["launches"] == w.nslices
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y))
    bsm.bsm_plan_debug(p, bsm.DEBUG_WITHHOLD_STAGE, 100_000_000)
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    bsm.bsm_plan_debug(p, bsm.DEBUG_NONE)
    bsm.bsm_device_status_clear()
    y.fill_(float("nan"))
    for _ in range(3):
        p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y))
    p.close()


def test_withheld_stage_in_a_group_launch_times_out_and_context_survives():
    """Rows split over groups of CTAs: the members of a group wait on one
    another too; with a stage withheld every wait still ends (timeout
    status), and the next execute is right."""
    import time
    import torch
    w = workload.uniform("fail group", workload.F32, 1, 19, 98304, 2.0, 0xFA12).materialize()
    x = to_device(w.x)
    y = torch.zeros_like(x)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_DYNAMIC)
    assert p.stats()["group_rows"] == 19          # 19 of the 25 groups of 6 CTAs on 152 SMs
    bsm.bsm_plan_debug(p, bsm.DEBUG_WITHHOLD_STAGE, 100_000_000)      # 0.1 s waits
    t0 = time.time()
    p.execute()
    torch.cuda.synchronize()
    assert time.time() - t0 < 5.0
    assert bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    bsm.bsm_plan_debug(p, bsm.DEBUG_NONE)
    bsm.bsm_device_status_clear()
    y.fill_(float("nan"))
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    check_all_against_oracle(w, to_host(y))
    p.close()


def test_corrupted_group_row_is_skipped_by_every_member():
    """A record of the group-row table pointing past the buffers: every
    member of the group that draws it skips it alike (no member waits for
    the others' partials), BSM_DEV_BOUNDS is set, and the other rows are
    right."""
    import torch
    w = workload.uniform("fail group corrupt", workload.F32, 1, 19, 98304, 2.0, 0xFA13).materialize()
    C = int(w.cols[0])
    x = to_device(w.x)
    sentinel = -7.0
    y = torch.full_like(x, sentinel)
    bsm.bsm_device_status_clear()
    p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, bsm.POLICY_RR)
    st = p.stats()
    assert st["group_rows"] == 19 and st["n_items"] == 19
    bsm.bsm_plan_debug(p, bsm.DEBUG_CORRUPT_PATCH, 7)         # the group table's slot 7
    p.execute()
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() & bsm.DEV_BOUNDS
    assert not bsm.bsm_device_status() & bsm.DEV_TIMEOUT
    yh = to_host(y).reshape(-1, C)
    untouched = np.all(yh == sentinel, axis=1)
    assert untouched.sum() == 1 and untouched[7]
    from oracle import softmax as O
    y64, _ = O.softmax_batched(w.x, w.offsets, w.rows, w.cols)
    ok = ~untouched
    assert np.max(np.abs(yh[ok].astype(np.float64) - y64.reshape(-1, C)[ok])) <= 2e-6
    p.close()
    bsm.bsm_device_status_clear()
