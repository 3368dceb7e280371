"""Rows longer than one shared-memory stage against the oracle, under every
policy, bit-identical across policies: forward rows split over groups of CTAs
(each CTA stages one part; the group exchanges (max, sum) partials), and the
paths that stream a row twice in chunks (a running max and rescaled sum,
then the output): few long rows cut into segments over two launches, and
the backward pass."""
import numpy as np
import pytest

from gpu_util import bits, check_all_against_oracle, run, to_device, to_host
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu

ALL = [bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR, bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF,
       bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX]


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    bsm.bsm_device_status_clear()


def _all(w, x):
    import torch
    ys = [run(w, x, p) for p in ALL]
    torch.cuda.synchronize()
    for y in ys[1:]:
        assert torch.equal(bits(y), bits(ys[0]))
    return ys[0]


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
def test_rows_just_over_and_far_over_a_stage(dtype):
    es = 4 if dtype == workload.F32 else 2
    limit = bsm.bsm_max_row_bytes() // es
    for B, R, C, flags in [(2, 3, limit + 16 // es, 0), (1, 2, 262144, 0),
                           (1, 1, 1 << 21, 0), (2, 5, 65536, workload.CAUSAL)]:
        w = workload.uniform("long", dtype, B, R, C, 4.0, 0x1046 + C + flags, flags).materialize()
        x = to_device(w.x)
        p = bsm.bsm_plan_create(x, x, w.rows, w.cols, dtype, bsm.POLICY_DYNAMIC, flags=flags)
        assert p.stats()["long_items"] == B * R
        p.close()
        y = _all(w, x)
        check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


def test_mixed_short_and_long_rows_in_one_batch():
    # ragged: 256 B .. 1.6 MB rows interleaved, some slices with one row
    rows = np.array([4, 1, 3, 2, 5, 1, 2], np.int32)
    cols = np.array([64, 400000, 2048, 120000, 512, 16, 70000], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.concatenate([[0], np.cumsum(sizes)[:-1]]).astype(np.int64)
    w = workload.Workload("mixed long", workload.F32, rows, cols, off, 0, 0x4D17, 3.0)
    w.materialize()
    x = to_device(w.x)
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))


def test_non_finite_long_rows():
    C = 100000
    rows = []
    rng = np.random.default_rng(3)
    for kind in range(4):
        r = rng.normal(0, 3, C).astype(np.float32)
        if kind == 1:
            r[77777] = np.nan
        elif kind == 2:
            r[5] = np.inf
        elif kind == 3:
            r[:] = -np.inf
            r[99999] = 1.0
        rows.append(r)
    w = workload.uniform("long nonfinite", workload.F32, 1, 4, C, 1.0, 0)
    w.x = np.stack(rows).reshape(-1)
    x = to_device(w.x)
    y = _all(w, x)
    yh = to_host(y).reshape(4, C)
    assert np.isnan(yh[1]).all() and np.isnan(yh[2]).all()
    assert yh[3, 99999] == 1.0 and np.count_nonzero(yh[3]) == 1
    check_all_against_oracle(w, to_host(y))


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
def test_many_long_rows_stream_whole_rows_in_one_launch(dtype):
    """With at least two waves of rows too short for a group each row is one
    segment that one CTA streams in a single launch (fewer rows are cut into
    segments over two launches).  Rows just over the cap get three stages of
    half a row: a row (two chunks) stays staged for its second pass.  Against
    the oracle, all policies bit-identical."""
    import torch
    es = 4 if dtype == workload.F32 else 2
    limit = bsm.bsm_max_row_bytes() // es
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    R, C = 2 * n_sm + 8, limit + 16 // es
    w = workload.uniform("many long", dtype, 1, R, C, 3.0, 0x10A6 + dtype).materialize()
    x = to_device(w.x)
    p = bsm.bsm_plan_create(x, x, w.rows, w.cols, dtype, bsm.POLICY_DYNAMIC)
    st = p.stats()
    assert st["long_items"] == R and st["launches"] == 1 and st["n_items"] == R
    assert st["group_rows"] == 0
    assert st["n_stages"] == 3 and 2 * st["stage_bytes"] >= C * es
    p.close()
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


def test_few_long_rows_are_segmented_over_two_launches():
    import torch
    es = 4
    limit = bsm.bsm_max_row_bytes() // es
    w = workload.uniform("few long", workload.F32, 1, 3, 8 * limit, 2.0, 0x5E6).materialize()
    x = to_device(w.x)
    p = bsm.bsm_plan_create(x, torch.empty_like(x), w.rows, w.cols, workload.F32, bsm.POLICY_DYNAMIC)
    st = p.stats()
    assert st["long_items"] == 3 and st["launches"] == 2 and st["n_items"] > 3
    p.close()
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
@pytest.mark.parametrize("chunks,flags", [(3, workload.CAUSAL), (4, 0)])
def test_many_long_rows_of_several_chunks(dtype, chunks, flags):
    """Two waves of rows of three and four stages' length: the three-chunk
    rows (four parts of 64 KiB at most: too few for a group) are streamed
    whole by one CTA each, starting the second pass on the chunk still
    staged and running backwards; the four-chunk rows go to groups of eight
    CTAs.  Under the causal mask most of every row is masked (the row index is
    below the column count)."""
    import torch
    es = 4 if dtype == workload.F32 else 2
    limit = bsm.bsm_max_row_bytes() // es
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    R, C = 2 * n_sm + 3, (chunks - 1) * limit + 16 // es * 7
    w = workload.uniform("many long %d" % chunks, dtype, 1, R, C, 3.0, 0x10B0 + chunks + dtype,
                         flags).materialize()
    x = to_device(w.x)
    p = bsm.bsm_plan_create(x, x, w.rows, w.cols, dtype, bsm.POLICY_DYNAMIC, flags=flags)
    st = p.stats()
    assert st["long_items"] == R and st["launches"] == 1
    assert st["group_rows"] == (0 if chunks == 3 else R)
    p.close()
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


# rows over groups: (rows, row length, dtype, group size on 152 SMs) -- one
# full wave each (as many rows as groups, n_sm // K)
GROUP_CASES = [(25, 98304, workload.F32, 6), (9, 262144, workload.F32, 16),
               (4, 524288, workload.F32, 32), (19, 262144, workload.BF16, 8),
               (9, 524288, workload.BF16, 16), (4, 1048576, workload.BF16, 32)]


@pytest.mark.parametrize("case", range(len(GROUP_CASES)))
@pytest.mark.parametrize("flags", [0, workload.CAUSAL])
def test_group_rows_every_group_size(case, flags):
    import torch
    R, C, dtype, k = GROUP_CASES[case]
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    w = workload.uniform("group rows", dtype, 1, R, C, 3.0, 0x6A0 + case + flags, flags).materialize()
    x = to_device(w.x)
    p = bsm.bsm_plan_create(x, torch.empty_like(x), w.rows, w.cols, dtype, bsm.POLICY_DYNAMIC,
                            flags=flags)
    st = p.stats()
    p.close()
    if n_sm == 152:
        assert st["group_k"] == k
    assert st["group_rows"] == R and st["launches"] == 1
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


def test_group_rows_beside_short_rows_two_launches():
    """A ragged batch: short rows (one launch of the regular kernel) and a
    wave of rows split over groups (a second, cooperative launch), slices
    interleaved and not contiguous."""
    rows = np.array([3, 20, 5, 19, 1, 0, 7], np.int32)
    cols = np.array([512, 200000, 64, 180000, 4096, 64, 2048], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.concatenate([[0], np.cumsum(sizes + 64)[:-1]]).astype(np.int64)
    w = workload.Workload("group mix", workload.F32, rows, cols, off, 0, 0x6B0, 3.0)
    w.materialize()
    import torch
    x = to_device(w.x)
    p = bsm.bsm_plan_create(x, torch.empty_like(x), w.rows, w.cols, workload.F32,
                            bsm.POLICY_DYNAMIC, offsets=w.offsets)
    st = p.stats()
    p.close()
    assert st["group_rows"] == 39 and st["launches"] == 2
    y = _all(w, x)
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


def test_non_finite_group_rows():
    """NaN, +inf, a row all -inf but one element and a row all -inf, inside
    a wave of rows split over groups: the same results as the definition."""
    C, R = 100000, 19
    rng = np.random.default_rng(5)
    x = rng.normal(0, 3, (R, C)).astype(np.float32)
    x[1, 77777] = np.nan
    x[2, 5] = np.inf
    x[3, :] = -np.inf
    x[3, 99999] = 1.0
    x[4, :] = -np.inf
    w = workload.uniform("group nonfinite", workload.F32, 1, R, C, 1.0, 0)
    w.x = x.reshape(-1)
    import torch
    xd = to_device(w.x)
    p = bsm.bsm_plan_create(xd, torch.empty_like(xd), w.rows, w.cols, workload.F32,
                            bsm.POLICY_DYNAMIC)
    assert p.stats()["group_rows"] == R
    p.close()
    y = _all(w, xd)
    yh = to_host(y).reshape(R, C)
    assert np.isnan(yh[1]).all() and np.isnan(yh[2]).all() and np.isnan(yh[4]).all()
    assert yh[3, 99999] == 1.0 and np.count_nonzero(yh[3]) == 1
    check_all_against_oracle(w, to_host(y))
