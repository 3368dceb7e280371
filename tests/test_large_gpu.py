"""Batches past 32-bit element (fp32) and byte (bf16) offsets: 4097 slices of
512 x 1024, 2^31 + 2^19 elements (8.6 GB per fp32 array, 4.3 GB per bf16
array).  Rows on both sides of element 2^31 (and, for bf16, of byte 2^32)
are checked against the oracle; the whole outputs of three policies must be
equal bit for bit.  The inputs are drawn on the device by torch (seeded) and
the sampled rows copied back for the oracle."""
import numpy as np
import pytest

from gpu_util import BF16_ULPS, FP32_TOL, bits, to_host
from oracle import softmax as O
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu

B, R, C = 4097, 512, 1024          # B * R * C = 2^31 + 2^19


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()


def _rows_to_check():
    """(slice, row) pairs: the first rows, the rows around element 2^31 and
    byte 2^32 of a bf16 array (the same element), and the last rows."""
    per_slice = R * C
    g = (1 << 31) // C                 # global row that starts at element 2^31
    picks = [0, 1, g - 2, g - 1, g, g + 1, B * R - 2, B * R - 1]
    return [(p // R, p % R) for p in picks] + [((1 << 31) // per_slice, 0)]


@pytest.mark.parametrize("dtype,flags", [(workload.F32, 0), (workload.BF16, workload.CAUSAL)])
def test_offsets_past_32_bits(dtype, flags):
    import torch
    tdt = torch.float32 if dtype == workload.F32 else torch.bfloat16
    n = B * R * C
    assert n > (1 << 31)
    gen = torch.Generator(device="cuda").manual_seed(0x2002070631 + dtype)
    x = (torch.randn(n, device="cuda", generator=gen) * 3.0).to(tdt)
    outs = []
    for pol in (bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF_LB, bsm.POLICY_RR):
        y = torch.empty_like(x)
        bsm.bsm_softmax_ex(x, y, B, R, C, dtype, pol, flags)
        torch.cuda.synchronize()
        outs.append(y)
        if len(outs) > 1:
            assert torch.equal(bits(outs[-1]), bits(outs[0])), bsm.POLICY_NAMES[pol]
            outs.pop()
    assert bsm.bsm_device_status() == 0
    y = outs[0]
    for s, r in _rows_to_check():
        a = (s * R + r) * C
        xr = to_host(x[a:a + C])
        yr = to_host(y[a:a + C])
        y64, yo = O.softmax_row(xr, r, flags)
        if dtype == workload.F32:
            assert float(np.max(np.abs(yr.astype(np.float64) - y64))) <= FP32_TOL, (s, r)
        else:
            d = np.abs(yr.astype(np.int32) - yo.astype(np.int32))
            assert int(d.max()) <= BF16_ULPS, (s, r)
    del x, y, outs
    torch.cuda.empty_cache()


@pytest.mark.parametrize("R_long,C_long", [(2049, 1 << 20), (9, 1 << 28)])
def test_long_rows_past_32_bits(R_long, C_long):
    """Rows longer than a stage past element 2^31: 2049 rows of 4 MiB (each
    row whole in one launch) and 9 rows of 1 GiB (segments over two
    launches); the rows on both sides of element 2^31 against the oracle."""
    import torch
    n = R_long * C_long
    assert n > (1 << 31)
    gen = torch.Generator(device="cuda").manual_seed(0x2002070632 + R_long)
    x = torch.randn(n, device="cuda", generator=gen) * 2.0
    y = torch.empty_like(x)
    bsm.bsm_softmax_ex(x, y, 1, R_long, C_long, workload.F32, bsm.POLICY_DYNAMIC, 0)
    y2 = torch.empty_like(x)
    bsm.bsm_softmax_ex(x, y2, 1, R_long, C_long, workload.F32, bsm.POLICY_RR, 0)
    torch.cuda.synchronize()
    assert torch.equal(bits(y), bits(y2))
    del y2
    assert bsm.bsm_device_status() == 0
    g = (1 << 31) // C_long
    for r in (g - 1, g, R_long - 1):
        a = r * C_long
        y64, _ = O.softmax_row(to_host(x[a:a + C_long]), r, 0)
        err = float(np.max(np.abs(to_host(y[a:a + C_long]).astype(np.float64) - y64)))
        assert err <= FP32_TOL, (r, err)
    del x, y
    torch.cuda.empty_cache()
