"""The schedule of real plans against the scheduling oracle, and a check of
the address -> die map the die-queue policies are built on.

Schedule: for CBMF (Sec. 4.1), CBMF_LB (Sec. 4.1 + 4.2) and MINIMAX (Sec. 4.2
general form), a plan is built on device buffers; the map it probed, its
patches (the host cutter's, checked against the device table), its SM
counts per die and its latency weights go into oracle/schedule_oracle.py,
which must give the same table counts, the same queues in the same order,
and the same moved patches.  The device table must hold, at every queue
slot, the record of the patch the queue names there.

Map: mapping a buffer twice gives (nearly) the same dies; the reads of the
die-check kernel (each die's SMs read the chunks mapped to it, or, inverted,
the others) cover the buffer exactly once -- the condition for its profiler
counters (how much traffic crossed dies) to mean something.
"""
import numpy as np
import pytest

from oracle import schedule_oracle as S
from paper_2002_07062_gb300 import bsm, workload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def setup():
    import torch
    import __graft_entry__ as g
    g.build()
    torch.cuda.set_device(0)
    yield
    bsm.bsm_cache_clear()


def _separable():
    t = bsm.bsm_topology_probe()
    if not t["separable"]:
        pytest.skip("this device's dies could not be told apart by the probe")
    return t


def _workloads():
    return [workload.uniform("sched fp32 96 x 512x512", workload.F32, 96, 512, 512, 1.0, 0x5C0),
            workload.ragged("sched ragged", workload.F32, 40, 1.0, 0x5C1)]


def _oracle_schedule(policy, patches, maps, cost, units, ln, lf, seed):
    table = S.bank_table(patches, maps, 2)
    bank = S.resolve_overlap(table, seed)
    L = S.counts(bank, 2)
    q = S.cbmf_queues(bank, 2)
    moved = []
    if policy == bsm.POLICY_CBMF_LB:
        r = S.load_balance(q, cost, units, ln, lf)
        q, moved = r.queues, r.moved
    elif policy == bsm.POLICY_MINIMAX:
        q, _ = S.minimax_lpt(table, units, ln, lf)
    return table, L, q, moved


@pytest.mark.parametrize("policy", [bsm.POLICY_CBMF, bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX])
@pytest.mark.parametrize("wi", [0, 1])
def test_device_plan_schedule_matches_oracle(policy, wi):
    import torch
    topo = _separable()
    w = _workloads()[wi]
    n = w.numel
    x = torch.empty(n, device="cuda", dtype=torch.float32).normal_()
    y = torch.empty_like(x)
    plan = bsm.bsm_plan_create(x, y, w.rows, w.cols, w.dtype, policy, offsets=w.offsets)
    try:
        st = plan.stats()
        sc = bsm.bsm_plan_get_schedule(plan)
        table_dev = bsm.bsm_plan_device_table(plan, 0)
    finally:
        plan.close()
    assert sc["n_queues"] == 2 and sc["map_chunk_bytes"] >= 128
    # the planner's inputs are the topology's: SMs per die, latencies rounded
    assert sc["units"][:2] == [max(1, v) for v in topo["sm_per_die"][:2]]
    assert sc["l_near"] == max(1, round(topo["l_near"]))
    assert sc["l_far"] == max(1, round(topo["l_far"]))
    # the patches (slice order) as the host cutter makes them for this device
    props = torch.cuda.get_device_properties(0)
    smem = getattr(props, "shared_memory_per_block_optin", None)
    if smem is None:
        pytest.skip("torch does not report the opt-in shared memory")
    lay = bsm.bsm_plan_layout_host(w.rows, w.cols, w.dtype, policy, props.multi_processor_count,
                                   smem, offsets=w.offsets)
    p0 = lay["phase0"]
    assert len(p0) == st["n_items"] == sc["n_items"]
    es = 4
    lo = p0["elem_offset"].astype(np.int64) * es
    hi = (p0["elem_offset"].astype(np.int64)
          + p0["nrows"].astype(np.int64) * p0["cols"].astype(np.int64)) * es
    patches = list(zip(lo.tolist(), hi.tolist()))
    chunk = sc["map_chunk_bytes"]
    xmap = sc["x_map"].tolist()
    assert len(xmap) == (n * es + chunk - 1) // chunk
    maps = [S.BankMap(chunk, xmap)]
    if sc["count_output_bytes"]:
        maps.append(S.BankMap(chunk, sc["y_map"].tolist() if sc["y_map"] is not None else xmap))
    # the work of a patch: the bytes it moves (its input read, its output written)
    cost = [2 * (b - a) for a, b in patches]
    units = sc["units"][:2]
    table, L, queues, moved = _oracle_schedule(policy, patches, maps, cost, units, sc["l_near"],
                                               sc["l_far"], sc["tie_seed"])
    assert st["N"][:2] == table.N
    assert st["L"][:2] == L and sum(L) == len(patches)
    assert st["overlap_items"] == sum(table.overlap)
    q = sc["queue"]
    for d in range(2):
        b, ln = sc["queue_begin"][d], sc["queue_len"][d]
        assert q[b:b + ln].tolist() == queues[d], "queue of die %d" % d
    assert sorted(q.tolist()) == list(range(len(patches)))      # every patch queued once
    assert sc["moved"].tolist() == moved
    assert st["moved_items"] == len(moved)
    # the device table: slot k holds the record of patch queue[k]
    assert len(table_dev) == len(p0)
    assert np.array_equal(table_dev, p0[q])


def test_die_map_is_stable_and_the_check_reads_every_chunk_once():
    import torch
    topo = _separable()
    nbytes = 64 << 20
    g = torch.Generator(device="cuda").manual_seed(0xD1E)
    buf = torch.randint(-2**31, 2**31 - 1, (nbytes // 4,), device="cuda", dtype=torch.int32,
                        generator=g)
    chunk = 128
    m1 = bsm.bsm_addr_die_map(buf, nbytes, chunk)
    m2 = bsm.bsm_addr_die_map(buf, nbytes, chunk)
    agree = float(np.mean(m1 == m2))
    share0 = float(np.mean(m1 == 0))
    print("die map of %d MiB at %d B: die 0 holds %.4f, two probes agree on %.5f; "
          "granularity %d B" % (nbytes >> 20, chunk, share0, agree, topo["granularity"]))
    assert agree >= 0.85
    assert 0.3 <= share0 <= 0.7
    want = int(np.bitwise_xor.reduce(buf.cpu().numpy().view(np.uint32)))
    for invert in (False, True):
        got, ms = bsm.bsm_die_check_read(buf, nbytes, chunk, m1, invert=invert)
        assert got == want, "invert=%s: the reads did not cover the buffer once" % invert
        assert ms > 0
    assert bsm.bsm_device_status() == 0
