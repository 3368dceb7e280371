"""The host-only patch table (bsm_plan_layout_host, given this device's SM
count and opt-in shared memory) against the plans bsm_plan_create builds on
the device: the same stage size and count, patch count and long-row count."""
import pytest

from paper_2002_07062_gb300 import bsm

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)


CASES = [
    # rows, cols, dtype, policy, op
    ([512] * 384, [512] * 384, bsm.F32, bsm.POLICY_DYNAMIC, 0),
    ([512] * 384, [512] * 384, bsm.BF16, bsm.POLICY_RR, 0),
    ([32] * 4096, [128] * 4096, bsm.BF16, bsm.POLICY_DYNAMIC, 0),
    ([64], [1 << 20], bsm.F32, bsm.POLICY_DYNAMIC, 0),
    ([2048], [65536], bsm.BF16, bsm.POLICY_DYNAMIC, 0),
    ([512] * 8, [2048] * 8, bsm.F32, bsm.POLICY_DYNAMIC, bsm.OP_BACKWARD),
    ([5, 0, 300, 2, 17], [40000, 64, 512, 131072, 8192], bsm.F32, bsm.POLICY_RR, 0),
    ([5, 0, 300, 2, 17], [40000, 64, 512, 131072, 8192], bsm.F32, bsm.POLICY_WHOLE_GPU, 0),
]


@pytest.mark.parametrize("case", range(len(CASES)))
def test_layout_matches_device_plan(case):
    import torch
    rows, cols, dtype, policy, op = CASES[case]
    props = torch.cuda.get_device_properties(0)
    smem = getattr(props, "shared_memory_per_block_optin", None)
    if smem is None:
        pytest.skip("torch does not report the opt-in shared memory")
    n = sum(r * c for r, c in zip(rows, cols))
    tdt = torch.float32 if dtype == bsm.F32 else torch.bfloat16
    x = torch.empty(n, device="cuda", dtype=tdt)
    y = torch.empty_like(x)
    x2 = torch.empty_like(x) if op == bsm.OP_BACKWARD else None
    plan = bsm.bsm_plan_create(x, y, rows, cols, dtype, policy, op=op, x2=x2)
    try:
        st = plan.stats()
    finally:
        plan.close()
    L = bsm.bsm_plan_layout_host(rows, cols, dtype, policy, props.multi_processor_count, smem, op=op)
    assert st["stage_bytes"] == L["stage_bytes"]
    assert st["n_stages"] == L["n_stages"]
    assert st["n_items"] == len(L["phase0"])
    assert st["long_items"] == L["long_rows"]
    if policy != bsm.POLICY_WHOLE_GPU:
        assert st["launches"] == (0 if not len(L["phase0"]) else 1 + (len(L["phase1"]) > 0))
