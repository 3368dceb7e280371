"""bsm_softmax_host: host buffers in, host buffers out, copies overlapped in
chunks.  Must give exactly the bits of the device-buffer path."""
import numpy as np
import pytest

from gpu_util import bits, to_device
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("k", [2, 3])
def test_host_pipeline_matches_device_path(k):
    import torch
    w = workload.config(k).materialize()
    R, C = int(w.rows[0]), int(w.cols[0])
    x = to_device(w.x)
    y_dev = torch.empty_like(x)
    bsm.bsm_softmax_ex(x, y_dev, w.nslices, R, C, w.dtype, bsm.POLICY_DYNAMIC, w.flags)
    xp = x.cpu().pin_memory()
    yp = torch.empty_like(xp).pin_memory()
    s = torch.cuda.Stream()
    bsm.bsm_softmax_host(xp, yp, w.nslices, R, C, w.dtype, bsm.POLICY_DYNAMIC, w.flags, s)
    s.synchronize()
    assert torch.equal(bits(yp), bits(y_dev.cpu()))


def test_host_pipeline_ragged_tail_in_place_and_pageable():
    import torch
    # 339 slices of 96 x 1024 fp32 (384 KiB each): two chunks of 128 slices
    # and a tail of 83, so both staging buffers are reused and a copy-out
    # is always issued after the next chunk's copy-in and kernel
    w = workload.uniform("host tail", workload.F32, 339, 96, 1024, 2.0, 0x4057).materialize()
    x = to_device(w.x)
    y_dev = torch.empty_like(x)
    bsm.bsm_softmax(x, y_dev, w.nslices, 96, 1024, w.dtype, bsm.POLICY_RR)
    ref = y_dev.cpu().numpy()
    # pageable numpy buffers, in place
    buf = w.x.copy()
    bsm.bsm_softmax_host(buf, buf, w.nslices, 96, 1024, w.dtype, bsm.POLICY_RR)
    torch.cuda.synchronize()
    assert np.array_equal(buf.view(np.uint32), ref.view(np.uint32))
    # twice in a row into a fresh output
    out = np.empty_like(w.x)
    for _ in range(2):
        out[:] = 0
        bsm.bsm_softmax_host(w.x, out, w.nslices, 96, 1024, w.dtype, bsm.POLICY_DYNAMIC)
        torch.cuda.synchronize()
        assert np.array_equal(out.view(np.uint32), ref.view(np.uint32))
