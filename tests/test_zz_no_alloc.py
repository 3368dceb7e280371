"""bsm_softmax_noalloc: the entry point for callers that cannot allocate
device memory (code inside a pre-reserved pool or arena, or a path that
must not add the device-wide synchronisation of cudaMalloc/cudaFree).  Its
scratch is a fixed array inside the library instead of a plan's table.

This file is collected last on purpose, so that a run stopping at the first
failure has run every other test first; the GPU test passes both alone in a
fresh process and after the rest of the suite."""
import ctypes

import numpy as np
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


@pytest.mark.gpu
def test_noalloc_matches_the_planned_entry_point_twice():
    import torch
    from gpu_util import FP32_TOL, to_device
    torch.cuda.set_device(0)
    cases = [workload.uniform("noalloc fp32", workload.F32, 24, 96, 512, 3.0, 0xA11C0),
             workload.uniform("noalloc bf16 causal", workload.BF16, 7, 70, 384, 8.0, 0xA11C1,
                              workload.CAUSAL)]
    for w in cases:
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
            assert not torch.isnan(y).any(), (w.name, call)
            if w.dtype == workload.F32:
                err = float((y.double() - ref.double()).abs().max())
                assert err <= FP32_TOL, (w.name, call, err)
            else:
                gi = y.view(torch.int16).int()
                ri = ref.view(torch.int16).int()
                assert int((gi - ri).abs().max()) <= 1, (w.name, call)
