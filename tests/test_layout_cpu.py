"""The patch table of a plan, on the host (no GPU): the C++ cutter behind
bsm_plan_create, reached through bsm_plan_layout_host, against properties
checked here from the batch itself.  Sec. 4 cuts a batch into patches (blocks
of consecutive rows); every row must then run exactly once, each patch must
fit a shared-memory stage, a row longer than a stage must be covered by its
segments exactly once, and the two launches of segmented rows must hold the
same segments; a row split over a group of CTAs must be one record whose
parts fit a stage of the group launch.  Worked figures: workload 2
(384 x 512 x 512 fp32) is 6144 patches of 32 rows in three 64 KiB stages; 64
rows of 4 MiB fp32 are 1216 segments over two launches; 256 rows of 1 MiB
fp32 go to eight groups of 19 CTAs."""
import random
from collections import Counter

import pytest

from paper_2002_07062_gb300 import bsm

SMEM = 232448            # opt-in shared memory per block of a GB300 SM (227 KiB)
HEADER = 1024            # barriers and stage metadata at the front of it
MIN_STAGE = 64 * 1024
MAX_STAGES = 8
QUEUE_POLICIES = (bsm.POLICY_DYNAMIC, bsm.POLICY_CBMF, bsm.POLICY_CBMF_LB, bsm.POLICY_MINIMAX)


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()


def _slices(rows, cols, offsets):
    out, pos = [], 0
    for s, (R, C) in enumerate(zip(rows, cols)):
        off = pos if offsets is None else offsets[s]
        out.append((off, R, C))
        pos = off + R * C
    return out


def check_layout(rows, cols, dtype, policy, n_sm=152, smem=SMEM, offsets=None, rows_per_item=0, op=0):
    es = 4 if dtype == bsm.F32 else 2
    vec = 16 // es
    ins = 2 if op == bsm.OP_BACKWARD else 1
    L = bsm.bsm_plan_layout_host(rows, cols, dtype, policy, n_sm, smem, offsets=offsets,
                                 rows_per_item=rows_per_item, op=op)
    stage, n_stages = L["stage_bytes"], L["n_stages"]
    avail = smem - HEADER
    assert stage % 128 == 0 and stage >= MIN_STAGE
    assert n_stages == min(MAX_STAGES, avail // stage) and n_stages >= 2

    sl = _slices(rows, cols, offsets)
    row_owner = {}                                 # element offset of a row -> (slice, row)
    for s, (off, R, C) in enumerate(sl):
        for r in range(R):
            row_owner[off + r * C] = (s, r)
    # a row that fits half the shared memory (with its partner row, for the
    # backward pass) is staged whole: never long
    whole_cap = (((avail // 2) & ~127) // ins) & ~127

    # rows split over groups of K CTAs (forward only): one record each, last
    # in phase 0, part_count = -K; they are all the rows longer than a stage
    # of their own, each part fits a third of the shared memory (three
    # stages), and the groups' waves are at least two thirds full
    K = L["group_k"]
    grp = [p for p in L["phase0"] if int(p["part_count"]) < 0]
    group_rows = set()
    if grp:
        assert op == 0 and 2 <= K <= min(n_sm, 128)
        assert all(int(p["part_count"]) < 0 for p in L["phase0"][len(L["phase0"]) - len(grp):])
        for p in grp:
            off, C, n, r0, R = (int(p[k]) for k in ("elem_offset", "cols", "nrows", "row0", "slice_rows"))
            assert int(p["part_count"]) == -K and n == 1 and int(p["col0"]) == 0
            assert off in row_owner and off not in group_rows
            s, r = row_owner[off]
            assert (r, R, C) == (r0, sl[s][1], sl[s][2])
            part = -(-(-(-C // K)) // vec) * vec      # ceil(C / K), whole vectors
            assert part * es <= (avail // 3) & ~127
            group_rows.add(off)
        assert group_rows == {o for o, (s, _) in row_owner.items() if sl[s][2] * es > whole_cap}
        G = n_sm // K
        waves = -(-len(grp) // G)
        assert 3 * len(grp) >= 2 * waves * G
    else:
        assert K == 0

    long_rows = set()
    for s, (off, R, C) in enumerate(sl):
        for r in range(R):
            if C * es * ins > stage and off + r * C not in group_rows:
                long_rows.add(off + r * C)
    assert all(C * es > whole_cap for (_, R, C) in sl if R > 0 and C * es * ins > stage)
    assert L["long_rows"] == len(long_rows) + len(group_rows)
    n_short = len(row_owner) - len(long_rows) - len(group_rows)

    seen = Counter()
    segs = {}                                      # long row -> [(col0, cols, part_count)]
    for p in L["phase0"]:
        if int(p["part_count"]) < 0:
            continue                               # a group row, checked above
        off, C, n, r0, R = (int(p[k]) for k in ("elem_offset", "cols", "nrows", "row0", "slice_rows"))
        assert n >= 1 and 0 <= r0 < R
        first = off - int(p["col0"])
        assert first in row_owner, off
        s, r = row_owner[first]
        assert r == r0 and sl[s][1] == R           # row0 and R name the first row's slice
        if int(p["part_count"]) > 0:               # a segment of a long row
            assert first in long_rows and n == 1
            assert 0 <= int(p["col0"]) and int(p["col0"]) + C <= sl[s][2]
            segs.setdefault(first, []).append((int(p["col0"]), C, int(p["part_count"])))
            continue
        assert int(p["col0"]) == 0
        assert n * C * es * ins <= stage           # the patch fits one stage
        if rows_per_item:
            assert n <= rows_per_item
        if policy == bsm.POLICY_WHOLE_GPU:
            assert n <= -(-R // n_sm)
        if policy in QUEUE_POLICIES:
            assert n <= max(1, -(-n_short // n_sm))
        if policy not in QUEUE_POLICIES:
            assert r0 + n <= R                     # RR / WHOLE_GPU: inside its slice
        for k in range(n):
            row = off + k * C
            assert row in row_owner and row not in long_rows and row not in group_rows, (off, k)
            assert sl[row_owner[row][0]][2] == C   # rows of one patch share a length
            seen[row] += 1
    short_rows = [o for o in row_owner if o not in long_rows and o not in group_rows]
    assert set(seen) == set(short_rows) and all(v == 1 for v in seen.values())

    # long rows: segments cover [0, C) once; every segment carries its row's count
    assert set(segs) == long_rows
    chunk = stage // ins // es
    multi = Counter()
    for first, parts in segs.items():
        C = sl[row_owner[first][0]][2]
        parts.sort()
        assert parts[0][0] == 0 and sum(c for _, c, _ in parts) == C
        assert all(a[0] + a[1] == b[0] for a, b in zip(parts, parts[1:]))
        assert all(pc == len(parts) for _, _, pc in parts)
        assert all(c0 % chunk == 0 for c0, _, _ in parts)     # whole chunks
        if len(parts) > 1:
            for c0, c, _ in parts:
                multi[(first + c0, c)] += 1
    # the second launch holds exactly the segments of rows cut into several
    got1 = Counter((int(p["elem_offset"]), int(p["cols"])) for p in L["phase1"])
    assert got1 == multi
    assert all(int(p["part_count"]) > 1 and int(p["nrows"]) == 1 for p in L["phase1"])
    if len(long_rows) >= 2 * n_sm:
        assert not multi                           # enough rows: each whole in one launch
    return L


def test_workload2_six_thousand_patches_of_32_rows():
    L = check_layout([512] * 384, [512] * 384, bsm.F32, bsm.POLICY_DYNAMIC)
    assert (L["stage_bytes"], L["n_stages"]) == (65536, 3)
    assert len(L["phase0"]) == 6144 and set(L["phase0"]["nrows"]) == {32}
    assert len(L["phase1"]) == 0


def test_four_mib_rows_are_1216_segments_over_two_launches():
    """64 fp32 rows of 4 MiB would need groups of 76 CTAs (too many to wait
    on): fewer rows than two per SM, so each is cut into 19 segments of whole
    chunks, 1216 over two launches.  fp32 rows streamed in chunks get three
    stages of a third of the shared memory: (232448 - 1024) / 3 rounded down
    to 128 bytes = 77056."""
    L = check_layout([64], [1 << 20], bsm.F32, bsm.POLICY_DYNAMIC)
    assert L["group_k"] == 0
    assert (L["stage_bytes"], L["n_stages"]) == (77056, 3)
    assert len(L["phase0"]) == 1216 and len(L["phase1"]) == 1216   # 19 per row
    assert L["long_rows"] == 64


def test_one_row_of_a_group_size_is_cut_into_segments():
    """A single 1 MiB fp32 row would keep seven of the eight groups idle: it
    is cut into segments of whole chunks instead (two launches): 1 MiB in
    chunks of at most 77056 bytes is 14 chunks, one segment each."""
    L = check_layout([1], [262144], bsm.F32, bsm.POLICY_DYNAMIC)
    assert L["group_k"] == 0
    assert len(L["phase0"]) == len(L["phase1"]) == 14


def test_rows_of_two_chunks_stay_staged():
    """bf16 rows of 128 KiB (two parts: too few for a group): three stages of
    half a row (two chunks per row), each row one patch, whole in one launch."""
    L = check_layout([2048], [65536], bsm.BF16, bsm.POLICY_DYNAMIC)
    assert L["group_k"] == 0
    assert (L["stage_bytes"], L["n_stages"]) == (65536, 3)
    assert len(L["phase0"]) == 2048 and len(L["phase1"]) == 0
    assert set(L["phase0"]["part_count"]) == {1} and set(L["phase0"]["cols"]) == {65536}


@pytest.mark.parametrize("C,dtype,k", [(65536, bsm.F32, 0), (98304, bsm.F32, 6), (262144, bsm.F32, 16),
                                       (524288, bsm.F32, 32), (1048576, bsm.F32, 0),
                                       (65536, bsm.BF16, 0), (262144, bsm.BF16, 8),
                                       (524288, bsm.BF16, 16), (917504, bsm.BF16, 28),
                                       (1048576, bsm.BF16, 32), (2097152, bsm.BF16, 0)])
def test_long_rows_group_sizes(C, dtype, k):
    """256 MiB of long rows: rows of 5 to 32 parts of at most 64 KiB go to
    groups of K CTAs, the fewest whose parts fit (K = ceil(row / 64 KiB)),
    each CTA holding one part; shorter rows (256 KiB fp32, 128 KiB bf16) stay
    on one CTA per row, longer ones (4 MiB of either type) are streamed
    twice."""
    es = 4 if dtype == bsm.F32 else 2
    R = (256 << 20) // (C * es)
    L = check_layout([R], [C], dtype, bsm.POLICY_DYNAMIC)
    assert L["group_k"] == k
    if k:
        assert len(L["phase0"]) == R and len(L["phase1"]) == 0


def test_backward_long_rows_keep_one_cta_per_row():
    """The backward pass keeps its long-row paths (no groups)."""
    L = check_layout([2048], [65536], bsm.BF16, bsm.POLICY_DYNAMIC, op=bsm.OP_BACKWARD)
    assert L["group_k"] == 0 and L["long_rows"] == 2048


@pytest.mark.parametrize("policy", [bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR] + list(QUEUE_POLICIES))
def test_patches_never_cross_slices_under_rr_and_whole_gpu(policy):
    # patches of at most 16 rows, which do not divide 3001: the queue
    # policies' patches run on into the next slice of the same shape
    rows, cols = [3001, 3001, 3001, 7], [256, 256, 256, 256]
    L = check_layout(rows, cols, bsm.F32, policy, rows_per_item=16)
    spans = any(int(p["row0"]) + int(p["nrows"]) > int(p["slice_rows"]) for p in L["phase0"])
    assert spans == (policy in QUEUE_POLICIES)


def test_small_batches_spread_over_every_sm():
    """A batch of fewer stage-filling patches than SMs is cut into patches of
    ceil(rows / SMs) rows under the queue policies (whose short queues are
    claimed one patch at a time), so that every SM takes one patch."""
    L = check_layout([64] * 8, [64] * 8, bsm.F32, bsm.POLICY_DYNAMIC)     # 8 x 64 x 64
    assert len(L["phase0"]) == 128 and set(L["phase0"]["nrows"]) == {4}
    L = check_layout([64] * 8, [64] * 8, bsm.F32, bsm.POLICY_RR)          # one patch per slice
    assert len(L["phase0"]) == 8
    L = check_layout([512] * 8, [512] * 8, bsm.F32, bsm.POLICY_CBMF_LB)   # 4096 rows
    assert len(L["phase0"]) == 152 and max(L["phase0"]["nrows"]) == 27
    # from one stage-filling patch per SM on, nothing changes
    L = check_layout([512] * 10, [512] * 10, bsm.F32, bsm.POLICY_DYNAMIC)
    assert set(L["phase0"]["nrows"]) == {32}


def test_backward_stage_holds_two_rows():
    L = check_layout([512] * 8, [2048] * 8, bsm.F32, bsm.POLICY_DYNAMIC, op=bsm.OP_BACKWARD)
    assert all(int(p["nrows"]) * 2048 * 4 * 2 <= L["stage_bytes"] for p in L["phase0"])


def test_errors():
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_plan_layout_host([4], [64], bsm.F32, bsm.POLICY_DYNAMIC, 0, SMEM)
    assert e.value.status == bsm.ERR_INVALID_ARG
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_plan_layout_host([4], [64], bsm.F32, bsm.POLICY_DYNAMIC, 152, 1024)
    assert e.value.status == bsm.ERR_INVALID_ARG
    with pytest.raises(bsm.BsmError) as e:                   # fewer than two stages fit
        bsm.bsm_plan_layout_host([4], [64], bsm.F32, bsm.POLICY_DYNAMIC, 152, HEADER + 100000)
    assert e.value.status == bsm.ERR_UNSUPPORTED
    with pytest.raises(bsm.BsmError) as e:                   # 3 fp32 columns: 12-byte rows
        bsm.bsm_plan_layout_host([4], [3], bsm.F32, bsm.POLICY_DYNAMIC, 152, SMEM)
    assert e.value.status == bsm.ERR_MISALIGNED
    L = bsm.bsm_plan_layout_host([], [], bsm.F32, bsm.POLICY_DYNAMIC, 152, SMEM)
    assert len(L["phase0"]) == 0 and len(L["phase1"]) == 0


@pytest.mark.parametrize("trial", range(60))
def test_random_batches(trial):
    rng = random.Random(0x20020706 + trial)
    dtype = rng.choice([bsm.F32, bsm.BF16])
    es = 4 if dtype == bsm.F32 else 2
    vec = 16 // es
    op = bsm.OP_BACKWARD if rng.random() < 0.25 else 0
    policy = rng.choice([bsm.POLICY_WHOLE_GPU, bsm.POLICY_RR] + list(QUEUE_POLICIES))
    n_sm = rng.choice([1, 2, 7, 148, 152, 160])
    smem = rng.choice([SMEM, 166912, 101376 + 65536])
    n = rng.randrange(0, 40)
    rows, cols = [], []
    for _ in range(n):
        kind = rng.random()
        if kind < 0.15:
            R, C = 0, vec * rng.randrange(1, 64)
        elif kind < 0.3:                           # longer than a stage
            R, C = rng.randrange(1, 6), vec * rng.randrange(8192 // vec * 16 // es, 8 * 65536 // vec)
        else:
            R, C = rng.randrange(1, 300), vec * rng.randrange(1, 2048 // vec + 1)
        rows.append(R)
        cols.append(C)
    offsets = None
    if rng.random() < 0.5:
        offsets, pos = [], 0
        for R, C in zip(rows, cols):
            pos += vec * rng.choice([0, 0, 1, 4])
            offsets.append(pos)
            pos += R * C
    rpi = rng.choice([0, 0, 1, 16, 64])
    try:
        check_layout(rows, cols, dtype, policy, n_sm=n_sm, smem=smem, offsets=offsets,
                     rows_per_item=rpi, op=op)
    except bsm.BsmError as e:
        # only a device too small for two stages may refuse a valid batch
        assert e.status == bsm.ERR_UNSUPPORTED and smem - HEADER < 2 * MIN_STAGE * (2 if op else 1), e


def test_edge_cases():
    # only empty slices: no patches, the default stages
    L = bsm.bsm_plan_layout_host([0, 0], [64, 64], bsm.F32, bsm.POLICY_RR, 152, SMEM)
    assert len(L["phase0"]) == 0 and L["n_stages"] == 3
    # in place (x == y) is allowed, a partial overlap is not
    check_layout([4], [64], bsm.F32, bsm.POLICY_DYNAMIC)
    assert len(bsm.bsm_plan_layout_host([4], [64], bsm.F32, bsm.POLICY_DYNAMIC, 152, SMEM,
                                        x=1 << 40, y=1 << 40)["phase0"]) == 4   # a row each
    with pytest.raises(bsm.BsmError) as e:
        bsm.bsm_plan_layout_host([4], [64], bsm.F32, bsm.POLICY_DYNAMIC, 152, SMEM,
                                 x=1 << 40, y=(1 << 40) + 64)
    assert e.value.status == bsm.ERR_INVALID_ARG
    # three 8 MiB bf16 rows, backward: segments of one chunk (28928 elements,
    # half of the 113 KiB stage per array), 145 per row
    L = check_layout([3], [1 << 22], bsm.BF16, bsm.POLICY_DYNAMIC, op=bsm.OP_BACKWARD)
    assert len(L["phase0"]) == len(L["phase1"]) == 3 * 145
    assert set(L["phase1"]["part_count"]) == {145}


@pytest.mark.parametrize("rows,cols,dtype,op,stage,n_stages", [
    # fp32 rows of two chunks of the 113 KiB cap keep two stages of the cap
    (1638, 40960, bsm.F32, bsm.OP_FORWARD, 115712, 2),
    # longer fp32 rows: three stages of a third of the shared memory
    (1024, 65536, bsm.F32, bsm.OP_FORWARD, 77056, 3),
    # bf16 rows streamed in chunks keep two stages of the cap
    (1024, 131072, bsm.BF16, bsm.OP_FORWARD, 115712, 2),
    # backward rows streamed by one CTA each (two waves or more): three stages
    (1024, 65536, bsm.F32, bsm.OP_BACKWARD, 77056, 3),
    # backward rows cut into segments (fewer than two per SM): two of the cap
    (256, 262144, bsm.F32, bsm.OP_BACKWARD, 115712, 2),
])
def test_stage_size_of_streamed_rows(rows, cols, dtype, op, stage, n_stages):
    """The stages that rows longer than one stage are streamed through, by
    row length, dtype and pass (232448 bytes of shared memory, 152 SMs)."""
    L = check_layout([rows], [cols], dtype, bsm.POLICY_DYNAMIC, op=op)
    assert L["group_k"] == 0
    assert (L["stage_bytes"], L["n_stages"]) == (stage, n_stages)
