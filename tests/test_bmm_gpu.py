"""Parity of the tensor-core batched matrix product (Sec. 6, the paper's
second batch algorithm) with the double-precision oracle, under every
scheduling policy, through the C ABI."""
import numpy as np
import pytest

from oracle import bmm_oracle as O
from oracle.softmax import bf16_bits_to_float
from paper_2002_07062_gb300 import bsm, workload as W

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")
if not torch.cuda.is_available():
    pytest.skip("needs a GPU", allow_module_level=True)

ALL_POLICIES = list(bsm.POLICIES.values())


def _dev(bits: np.ndarray):
    return torch.from_numpy(bits.view(np.int16)).cuda()


def _run(w: W.BmmWorkload, a_bits, bt_bits, policy, B=None):
    B = w.B if B is None else B
    da, db = _dev(a_bits), _dev(bt_bits)
    dt = torch.float32 if w.out_dtype == W.F32 else torch.int16
    c = torch.full((B * w.M * w.N,), -1, dtype=dt, device="cuda")
    bsm.bsm_bmm(da, db, c, B, w.M, w.N, w.K, w.out_dtype, policy)
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0
    return c


def _host(c, w: W.BmmWorkload, B):
    h = c.cpu().numpy()
    if w.out_dtype == W.F32:
        return h.astype(np.float64).reshape(B, w.M, w.N)
    return bf16_bits_to_float(h.view(np.uint16)).astype(np.float64).reshape(B, w.M, w.N)


def _bound(w: W.BmmWorkload, a_bits, bt_bits, B):
    """fp32 accumulation of exact bf16 products: |c32 - c| <= (K + 2) u sum|a b|,
    u = 2^-24; a bf16 result adds half an ulp of the result (2^-8 relative)."""
    aa = np.abs(bf16_bits_to_float(a_bits).astype(np.float64)).reshape(B, w.M, w.K)
    bb = np.abs(bf16_bits_to_float(bt_bits).astype(np.float64)).reshape(B, w.N, w.K)
    absprod = np.matmul(aa, np.transpose(bb, (0, 2, 1)))
    return (w.K + 2) * 2.0 ** -24 * absprod


def _check(w, got, ref, eps):
    if w.out_dtype == W.F32:
        bad = np.abs(got - ref) > eps + 1e-30
    else:
        bad = np.abs(got - ref) > eps + 2.0 ** -8 * (np.abs(ref) + eps) + 1e-30
    assert not bad.any(), (int(bad.sum()), np.argwhere(bad)[:5])


SHAPES = [  # B, M, N, K: every tile width (N = 64, 128, 256 blocks), ragged tile counts
    (1, 128, 64, 64), (1, 128, 128, 64), (1, 128, 256, 64), (2, 256, 192, 128),
    (3, 384, 320, 192), (5, 128, 512, 512), (9, 256, 64, 1024),
]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("out", [W.F32, W.BF16])
def test_bmm_matches_oracle(shape, out):
    B, M, N, K = shape
    w = W.BmmWorkload("t", B, M, N, K, out, seed=7 + B + K, sigma=1.0)
    a, bt = w.operands()
    ref = O.bmm_f64(a, bt, B, M, N, K)
    eps = _bound(w, a, bt, B)
    got = _host(_run(w, a, bt, bsm.POLICY_DYNAMIC), w, B)
    _check(w, got, ref, eps)


@pytest.mark.parametrize("out", [W.F32, W.BF16])
def test_small_integer_operands_are_exact(out):
    """Integer operands in [-6, 6] with K = 256: every partial sum is an
    integer below 2^24, so fp32 accumulation is exact in any order and the
    result equals the oracle's correctly rounded one, bit for bit."""
    B, M, N, K = 4, 256, 128, 256
    w = W.BmmWorkload("int", B, M, N, K, out, seed=11, kind="int")
    a, bt = w.operands()
    ref = O.bmm_f64(a, bt, B, M, N, K)
    c = _run(w, a, bt, bsm.POLICY_DYNAMIC).cpu().numpy()
    if out == W.F32:
        assert np.array_equal(c.reshape(B, M, N), ref.astype(np.float32))
    else:
        assert np.array_equal(c.view(np.uint16).reshape(B, M, N), O.round_bf16(ref))


@pytest.mark.parametrize("out", [W.F32, W.BF16])
def test_every_policy_gives_the_same_bits(out):
    """Policies only move tiles between SMs; each tile is computed the same
    way, so all six schedules produce identical bits."""
    B, M, N, K = 24, 256, 256, 192
    w = W.BmmWorkload("pol", B, M, N, K, out, seed=3)
    a, bt = w.operands()
    outs = [_run(w, a, bt, p) for p in ALL_POLICIES]
    for p, c in zip(ALL_POLICIES[1:], outs[1:]):
        assert torch.equal(c, outs[0]), bsm.POLICY_NAMES[p]
    _check(w, _host(outs[0], w, B), O.bmm_f64(a, bt, B, M, N, K), _bound(w, a, bt, B))


@pytest.mark.parametrize("k", [1, 2])
def test_paper_shapes_sampled_slices(k):
    """The two batched products of Sec. 6 at full size (384 slices), run in
    the launch configuration the benchmark times; 12 slices (first, last and
    spread) compared element by element with the oracle; all six policies
    bit-identical on the whole output."""
    w = W.bmm_config(k)
    a, bt = w.operands()
    outs = {p: _run(w, a, bt, p) for p in ALL_POLICIES}
    first = outs[bsm.POLICY_DYNAMIC]
    for p, c in outs.items():
        assert torch.equal(c, first), bsm.POLICY_NAMES[p]
    got = _host(first, w, w.B)
    slices = sorted({0, w.B - 1, *np.random.default_rng(k).choice(w.B, 10, replace=False).tolist()})
    sa, sb = w.operands(slices)
    ref = O.bmm_f64(sa, sb, len(slices), w.M, w.N, w.K)
    _check(w, got[slices], ref, _bound(w, sa, sb, len(slices)))


def test_many_small_slices_and_repeated_launches():
    """4096 one-tile slices: the queue heads reset themselves between launches."""
    B, M, N, K = 4096, 128, 64, 64
    w = W.BmmWorkload("many", B, M, N, K, W.F32, seed=21)
    a, bt = w.operands()
    da, db = _dev(a), _dev(bt)
    c1 = torch.zeros(B * M * N, dtype=torch.float32, device="cuda")
    c2 = torch.zeros_like(c1)
    for p in (bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF_LB, bsm.POLICY_RR):
        for _ in range(3):
            bsm.bsm_bmm(da, db, c1, B, M, N, K, W.F32, p)
        bsm.bsm_bmm(da, db, c2, B, M, N, K, W.F32, p)
        torch.cuda.synchronize()
        assert torch.equal(c1, c2)
    assert bsm.bsm_device_status() == 0
    got = c1.cpu().numpy().astype(np.float64).reshape(B, M, N)
    idx = [0, 1, 2047, 4095]
    sa, sb = w.operands(idx)
    _check(w, got[idx], O.bmm_f64(sa, sb, len(idx), M, N, K), _bound(w, sa, sb, len(idx)))


def test_non_finite_inputs_propagate():
    """inf * 0 = NaN and inf + finite = inf, as in IEEE arithmetic."""
    B, M, N, K = 1, 128, 64, 64
    w = W.BmmWorkload("nf", B, M, N, K, W.F32, seed=5)
    a, bt = w.operands()
    a = a.copy()
    bt = bt.copy()
    a[3 * K + 5] = 0x7F80        # A[3, 5] = +inf
    bt[:] = 0x3F80               # Bt = 1.0 everywhere: row 3 of C = +inf
    a[7 * K:8 * K] = 0x0000      # A[7, :] = 0 ...
    bt[9 * K + 4] = 0x7F80       # ... times Bt[9, 4] = inf: C[7, 9] = NaN
    c = _host(_run(w, a, bt, bsm.POLICY_DYNAMIC), w, B)[0]
    assert np.isposinf(np.delete(c[3], 9)).all()   # column 9 also meets Bt's inf
    assert np.isnan(c[7, 9])
    assert np.isfinite(np.delete(c[7], 9)).all()


def test_shape_errors_and_empty_batches():
    dt = torch.int16
    a = torch.zeros(128 * 64, dtype=dt, device="cuda")
    c = torch.zeros(128 * 64, dtype=torch.float32, device="cuda")
    for (M, N, K) in [(64, 64, 64), (128, 32, 64), (128, 64, 48), (128, 64, 0)]:
        with pytest.raises(bsm.BsmError) as e:
            bsm.bsm_bmm(a, a, c, 1, M, N, K, W.F32, bsm.POLICY_DYNAMIC)
        assert e.value.status == bsm.ERR_UNSUPPORTED
    bsm.bsm_bmm(a, a, c, 0, 128, 64, 64, W.F32, bsm.POLICY_DYNAMIC)
    with pytest.raises(bsm.BsmError) as e:          # output overlaps an operand
        bsm.bsm_bmm(a, a, a, 1, 128, 64, 64, W.BF16, bsm.POLICY_DYNAMIC)
    assert e.value.status == bsm.ERR_INVALID_ARG
    torch.cuda.synchronize()
    assert bsm.bsm_device_status() == 0


@pytest.mark.parametrize("N", [64, 128, 256])
@pytest.mark.parametrize("extra", [5, 76 + 7])
@pytest.mark.parametrize("out", [W.F32, W.BF16])
def test_ragged_tile_counts_are_exact(N, extra, out):
    """Tile counts one or two waves plus a few over the SMs, every tile
    width: integer operands make every result exact, equal to the oracle and,
    bit for bit, between the dynamic and the round-robin schedules."""
    n_sm = torch.cuda.get_device_properties(0).multi_processor_count
    B, M, K = n_sm // 2 + extra, 256, 192
    w = W.BmmWorkload("ragged waves", B, M, N, K, out, seed=29 + N + extra, kind="int")
    a, bt = w.operands()
    ref = O.bmm_f64(a, bt, B, M, N, K)
    dyn = _run(w, a, bt, bsm.POLICY_DYNAMIC)
    rr = _run(w, a, bt, bsm.POLICY_RR)
    assert torch.equal(dyn, rr)
    c = dyn.cpu().numpy()
    if out == W.F32:
        assert np.array_equal(c.reshape(B, M, N), ref.astype(np.float32))
    else:
        assert np.array_equal(c.view(np.uint16).reshape(B, M, N), O.round_bf16(ref))
