"""GPU parity of the batched softmax (through the C ABI) against the
double-precision oracle, under every scheduling policy.

fp32 output: max |y - oracle| <= 2e-6.  bf16 output: within 1 bf16 ulp of
the oracle's round-to-nearest-even result.  Every policy must give the same
bits (one row routine, fixed reduction order), every row must be written,
and nothing outside y may be touched."""
import numpy as np
import pytest

from gpu_util import (bits, check_all_against_oracle, check_every_element_against_oracle, run,
                      to_device, to_host)
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
    yield
    bsm.bsm_cache_clear()


def _all_policies_identical(w, x, policies=ALL):
    import torch
    ys = [run(w, x, p) for p in policies]
    torch.cuda.synchronize()
    for p, y in zip(policies[1:], ys[1:]):
        assert torch.equal(bits(y), bits(ys[0])), "policy %d differs from %d" % (p, policies[0])
    return ys[0]


def _ragged_all_classes(dtype, flags, seed, nslices=24, col_steps=160):
    # C in 16-byte vectors: 1..col_steps (160: up to 2.5 KiB rows, the register
    # routines; 768: up to 12 KiB rows, the shared-memory routines); R 1..60
    unit = 4 if dtype == workload.F32 else 8
    return workload.ragged("classes", dtype, nslices, 2.0, seed, flags, row_unit=1,
                           row_steps=60, col_unit=unit, col_steps=col_steps).materialize()


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
@pytest.mark.parametrize("flags", [0, bsm.FLAG_CAUSAL])
@pytest.mark.parametrize("col_steps", [160, 768])
def test_ragged_every_row_routine_full_parity(dtype, flags, col_steps):
    w = _ragged_all_classes(dtype, flags, 100 + 2 * dtype + flags + col_steps, col_steps=col_steps)
    x = to_device(w.x)
    y = _all_policies_identical(w, x)
    check_all_against_oracle(w, to_host(y))
    assert bsm.bsm_device_status() == 0


def test_workload1_full_parity():
    w = workload.config(1).materialize()
    x = to_device(w.x)
    y = _all_policies_identical(w, x)
    check_all_against_oracle(w, to_host(y))


@pytest.mark.parametrize("k", [2, 3, 5])
def test_uniform_workloads_full_size(k):
    import torch
    w = workload.config(k).materialize()
    x = to_device(w.x)
    y = _all_policies_identical(w, x)
    yh = to_host(y)
    # every element against the oracle (the launch configuration the bench times)
    check_every_element_against_oracle(w, yh)
    R, C = int(w.rows[0]), int(w.cols[0])
    yd = y.view(-1, C).double()
    assert not torch.isnan(yd).any()                     # every row written
    s = yd.sum(dim=1)
    tol = C * 2.0 ** -24 * 4 if w.dtype == workload.F32 else 0.01
    assert float((s - 1).abs().max()) <= tol
    if w.flags & bsm.FLAG_CAUSAL:
        y3 = y.view(w.nslices, R, C)
        upper = torch.triu(torch.ones(R, C, dtype=torch.bool, device=y.device), diagonal=1)
        assert int((y3[:, upper] != 0).sum()) == 0        # masked entries exactly 0
        assert bool((y3[:, 0, 0] == 1).all())             # row 0 one-hot
    assert bsm.bsm_device_status() == 0


def test_ragged_workload4_full_size():
    import torch
    w = workload.config(4).materialize()
    x = to_device(w.x)
    y = _all_policies_identical(w, x, [bsm.POLICY_RR, bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF,
                                       bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX,
                                       bsm.POLICY_WHOLE_GPU])
    yh = to_host(y)
    check_every_element_against_oracle(w, yh)
    assert not torch.isnan(y).any()
    for s in range(0, w.nslices, 37):
        R, C = int(w.rows[s]), int(w.cols[s])
        a = int(w.offsets[s])
        ss = y[a:a + R * C].view(R, C).double().sum(dim=1)
        assert float((ss - 1).abs().max()) <= C * 2.0 ** -24 * 4
    assert bsm.bsm_device_status() == 0


def test_guard_bands_untouched_and_in_place():
    import torch
    w = _ragged_all_classes(workload.F32, 0, 9, nslices=10)
    x = to_device(w.x)
    pad = 4096
    big = torch.full((w.numel + 2 * pad,), 1234.5, dtype=torch.float32, device="cuda")
    y = big[pad:pad + w.numel]
    run(w, x, bsm.POLICY_DYNAMIC, y=y)
    torch.cuda.synchronize()
    assert bool((big[:pad] == 1234.5).all()) and bool((big[pad + w.numel:] == 1234.5).all())
    ref = to_host(y)
    check_all_against_oracle(w, ref)
    # in place: x == y gives the same bits
    xi = x.clone()
    run(w, xi, bsm.POLICY_CBMF_LB, y=xi)
    torch.cuda.synchronize()
    assert np.array_equal(to_host(xi).view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
def test_longest_row_and_single_row(dtype):
    es = 4 if dtype == workload.F32 else 2
    cmax = bsm.bsm_max_row_bytes() // es
    for R, C in [(3, cmax), (1, 16 // es), (1, cmax), (2, 16 // es * 3)]:
        w = workload.uniform("edge", dtype, 2, R, C, 3.0, 77 + C).materialize()
        x = to_device(w.x)
        y = _all_policies_identical(w, x)
        check_all_against_oracle(w, to_host(y))


def test_non_finite_rows_match_oracle():
    C = 64
    rows = []
    rng = np.random.default_rng(1)
    for kind in range(6):
        r = rng.normal(0, 2, C).astype(np.float32)
        if kind == 1:
            r[5] = np.nan
        elif kind == 2:
            r[9] = np.inf
        elif kind == 3:
            r[:] = -np.inf
        elif kind == 4:
            r[:] = -np.inf
            r[3] = 1.0
        elif kind == 5:
            r[:] = -np.inf
            r[3] = r[40] = 2.0
        rows.append(r)
    xs = np.stack(rows).reshape(-1)
    w = workload.uniform("nonfinite", workload.F32, 1, len(rows), C, 1.0, 0)
    w.x = xs
    x = to_device(xs)
    y = _all_policies_identical(w, x)
    yh = to_host(y).reshape(-1, C)
    assert np.isnan(yh[1]).all() and np.isnan(yh[2]).all() and np.isnan(yh[3]).all()
    assert yh[4, 3] == 1.0 and np.count_nonzero(yh[4]) == 1
    assert yh[5, 3] == 0.5 and yh[5, 40] == 0.5 and np.count_nonzero(yh[5]) == 2
    check_all_against_oracle(w, to_host(y))


@pytest.mark.parametrize("C", [512, 128])
def test_causal_bf16_non_finite_in_masked_and_unmasked_positions(C):
    """Causal bf16 rows: a NaN or +inf in a masked position turns the row into
    NaN (NaN + (-inf), +inf + (-inf)), whether its vector is masked for every
    lane of the warp (no exponential is taken there), straddles the diagonal,
    or is unmasked; a -inf in a masked position changes nothing."""
    from oracle import softmax as O
    R = 8
    rng = np.random.default_rng(C)
    x = rng.normal(0, 3, (R, C)).astype(np.float32)
    x[1, C - 12] = np.nan            # far right of row 1: warp-wide masked vector
    x[2, 3] = np.inf                 # just past the diagonal of row 2
    x[3, C // 2:C // 2 + 40] = -np.inf   # masked -inf: no effect
    x[4, C // 3:C // 3 + 60] = -np.inf
    x[4, 2] = np.inf                 # unmasked +inf
    x[5, 5] = np.nan                 # on the diagonal (unmasked)
    x[6, 7:] = np.nan                # everything masked is NaN
    bits16 = (x.view(np.uint32) >> 16).astype(np.uint16)   # exact: the draws are re-read as bf16
    bits16[np.isnan(x)] = 0x7FC0
    w = workload.uniform("causal nonfinite", workload.BF16, 3, R, C, 1.0, 0, workload.CAUSAL)
    w.x = np.tile(bits16.reshape(-1), 3)
    xd = to_device(w.x)
    y = _all_policies_identical(w, xd)
    yh = to_host(y).reshape(3, R, C)
    _, yr = O.softmax_batched(w.x, w.offsets, w.rows, w.cols, w.flags)
    yr = yr.reshape(3, R, C)
    nan_g = (yh & 0x7FFF) > 0x7F80
    nan_o = (yr & 0x7FFF) > 0x7F80
    assert np.array_equal(nan_g, nan_o)
    for s in range(3):
        for r in (1, 2, 4, 5, 6):
            assert nan_g[s, r].all(), (s, r)
        for r in (0, 3, 7):
            assert not nan_g[s, r].any(), (s, r)
    ok = ~nan_o
    assert np.max(np.abs(yh[ok].astype(np.int32) - yr[ok].astype(np.int32))) <= 1
    assert bsm.bsm_device_status() == 0


def test_argument_errors_on_device():
    import torch
    x = torch.zeros(4 * 64 + 8, device="cuda")
    y = torch.zeros_like(x)
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_softmax(x.data_ptr() + 4, y, 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    assert e.value.status == bsm.ERR_MISALIGNED
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_softmax(x, y, 1, 1, 6, bsm.F32, bsm.POLICY_RR)          # 24-byte rows
    assert e.value.status == bsm.ERR_MISALIGNED
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_softmax(x, x.data_ptr() + 16, 4, 1, 64, bsm.F32, bsm.POLICY_RR)
    assert e.value.status == bsm.ERR_INVALID_ARG                        # partial overlap
    # a backward row longer than half a stage streams in chunks (no limit):
    # y = 1/C everywhere and dy = 1 give dx = 1/C * (1 - 1) = 0 exactly
    big = bsm.bsm_max_row_bytes() // 8 + 4
    yb = torch.full((big,), 1.0 / 1024, device="cuda")
    gb = torch.ones(big, device="cuda")
    db = torch.full((big,), float("nan"), device="cuda")
    bsm.bsm_softmax_backward(yb, gb, db, 1, 1, big, bsm.F32, bsm.POLICY_RR)
    torch.cuda.synchronize()
    dot = (big / 1024.0)
    assert torch.all(db == torch.tensor(1.0 / 1024, device="cuda") * (1.0 - dot))
    with pytest.raises(bsm.BsmError) as e:                              # overlapping slices
        bsm.bsm_softmax_ragged(x, y, [0, 32], [1, 1], [64, 64], bsm.F32, bsm.POLICY_RR)
    assert e.value.status == bsm.ERR_INVALID_ARG
    assert bsm.bsm_device_status() == 0


def test_topology_and_plan_stats():
    import torch
    t = bsm.bsm_topology_probe()
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    assert t["n_sm"] == n_sm
    seen = [d for d in t["sm_die"] if d >= 0]
    assert len(seen) >= n_sm * 0.9
    assert t["l_near"] > 0 and t["l_far"] >= t["l_near"]
    assert sum(t["sm_per_die"]) == len(seen)
    w = workload.config(2)
    x = torch.empty(w.numel, device="cuda")
    y = torch.empty_like(x)
    for pol in (bsm.POLICY_CBMF, bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX):
        p = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, pol)
        st = p.stats()
        n = st["n_items"]
        assert sum(st["L"][:st["n_die"]]) == n                         # sum L = N
        assert sum(st["N"][:st["n_die"]]) >= n                         # sum N >= N
        assert sum(st["queue_items"][:st["n_die"]]) == n
        p.close()


@pytest.mark.parametrize("dtype", [workload.F32, workload.BF16])
def test_ragged_batch_with_empty_slices(dtype):
    """Zero-row slices anywhere in a ragged batch (first, between same-shape
    slices, before a long row, last) are skipped; the other slices match the
    oracle and every policy gives the same bits; elements outside the slices
    (a gap) keep their sentinel."""
    import torch
    es = 4 if dtype == workload.F32 else 2
    long_c = bsm.bsm_max_row_bytes() // es + 16 // es
    rows = np.array([0, 3, 0, 3, 5, 0, 2, 1, 0], np.int32)
    cols = np.array([64, 128, 128, 128, 256, long_c, long_c, 512, 64], np.int32)
    sizes = rows.astype(np.int64) * cols
    off = np.zeros(len(rows), np.int64)
    pos = 0
    for i in range(len(rows)):
        off[i] = pos
        pos += int(sizes[i]) + (64 if i == 4 else 0)      # a gap after slice 4
    w = workload.Workload("empty slices", dtype, rows, cols, off, 0, 0xE3B7, 2.0)
    w.x = workload.fill_normal(pos, dtype, w.seed, w.sigma)
    x = to_device(w.x)
    outs = []
    for pol in (bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR, bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF,
                bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX):
        y = torch.full_like(x, -7.0)
        bsm.bsm_softmax_ragged(x, y, w.offsets, w.rows, w.cols, dtype, pol)
        outs.append(y)
    torch.cuda.synchronize()
    for y in outs[1:]:
        assert torch.equal(bits(y), bits(outs[0]))
    yh = to_host(outs[0])
    gap = slice(int(off[4] + sizes[4]), int(off[4] + sizes[4]) + 64)
    sentinel = to_host(torch.full((1,), -7.0, dtype=x.dtype, device="cuda"))[0]
    assert np.all(yh[gap] == sentinel)
    check_all_against_oracle(w, yh)
    assert bsm.bsm_device_status() == 0
