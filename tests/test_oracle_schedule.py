"""Pins of the scheduling oracle (Sec. 4.1 Cluster Beamforming, Sec. 4.2 Load
balancing) against the paper's printed table, its stated equalities and
inequalities, a published generator test vector and brute-force optimisation."""
import json
import os
import random

import pytest

from oracle import schedule_oracle as S

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_splitmix64_published_vector():
    lines = [l for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt"))
             if l.strip() and not l.startswith("#")]
    want = [int(l, 16) for l in lines]
    assert [S.splitmix64(0, i) for i in range(3)] == want


def test_paper_batch_to_bank_table():
    g = json.load(open(os.path.join(GOLDEN, "batch_bank_table.json")))
    m = S.BankMap(g["chunk"], g["bank_of_chunk"])
    t = S.bank_table([tuple(p) for p in g["patches"]], [m], 4)
    presence = [[1 if v > 0 else 0 for v in row] for row in t.bytes_on_bank]
    assert presence == g["table"]
    assert t.overlap == g["overlap"]
    assert t.N == g["N"]
    n = len(g["patches"])
    assert sum(t.N) > n                        # N_x + N_y + N_z + N_w > N
    bank = S.resolve_overlap(t, tie_seed=1)
    assert bank == g["resolved_bank"]
    L = S.counts(bank, 4)
    assert L == g["L"] and sum(L) == n         # L_x + L_y + L_z + L_w = N


def test_sum_N_equals_N_without_overlap():
    m = S.BankMap(1024, [0, 1] * 8)
    patches = [(k * 1024, (k + 1) * 1024) for k in range(16)]
    t = S.bank_table(patches, [m], 2)
    assert sum(t.overlap) == 0 and sum(t.N) == 16
    bank = S.resolve_overlap(t, 0)
    assert bank == [0, 1] * 8
    assert S.cbmf_queues(bank, 2) == [list(range(0, 16, 2)), list(range(1, 16, 2))]


def test_majority_rule_and_output_bytes_count():
    m = S.BankMap(256, [0, 1, 1, 1])
    t = S.bank_table([(0, 1024)], [m], 2)
    assert t.bytes_on_bank == [[256, 768]] and t.overlap == [1]
    assert S.resolve_overlap(t, 123) == [1]
    # input on bank 0, output on bank 1, more output bytes on bank 1 -> bank 1
    mx = S.BankMap(256, [0, 0, 0, 0])
    my = S.BankMap(256, [1, 1, 1, 0])
    t = S.bank_table([(0, 1024)], [mx, my], 2)
    assert t.bytes_on_bank == [[1280, 768]]
    assert S.resolve_overlap(t, 5) == [0]
    # partial chunks are counted by the byte
    t = S.bank_table([(100, 300)], [S.BankMap(256, [0, 1])], 2)
    assert t.bytes_on_bank == [[156, 44]]


def test_ties_are_fair_coins():
    n = 4000
    m = S.BankMap(128, [0, 1] * n)
    patches = [(k * 256, (k + 1) * 256) for k in range(n)]
    t = S.bank_table(patches, [m], 2)
    assert all(row == [128, 128] for row in t.bytes_on_bank)
    bank = S.resolve_overlap(t, tie_seed=0xC0FFEE)
    ones = sum(bank)
    assert abs(ones - n / 2) < 4 * (n ** 0.5) / 2          # within 4 sigma
    # reproducible for a seed, different for another
    assert bank == S.resolve_overlap(t, tie_seed=0xC0FFEE)
    assert bank != S.resolve_overlap(t, tie_seed=0xC0FFEF)


def test_three_way_ties_cover_all_banks():
    n = 3000
    m = S.BankMap(64, [0, 1, 2] * n)
    patches = [(k * 192, (k + 1) * 192) for k in range(n)]
    bank = S.resolve_overlap(S.bank_table(patches, [m], 3), 77)
    for b in range(3):
        assert abs(bank.count(b) - n / 3) < 4 * (n * (1 / 3) * (2 / 3)) ** 0.5


def test_load_balance_fixes_the_first_portion_degenerate_map():
    """Sec. 4.2: every patch judged by its first portion lands on one bank; LB
    must spread it back out."""
    n = 64
    cost = [1000] * n
    queues = [list(range(n)), []]
    out = S.load_balance(queues, cost, units=[76, 76], l_near=1, l_far=1)
    assert sorted(out.queues[0] + out.queues[1]) == list(range(n))
    assert len(out.queues[0]) == 32 and len(out.queues[1]) == 32
    assert out.moved == list(range(63, 31, -1))            # last natives first


def test_weighted_split_is_inverse_to_latency():
    n = 300
    cost = [10] * n
    out = S.load_balance([list(range(n)), []], cost, units=[1, 1], l_near=1, l_far=2)
    far = sum(cost[i] for i in out.queues[1])
    near = sum(cost[i] for i in out.queues[0])
    # near : far bytes = l_far : l_near = 2 : 1, to within one patch
    assert abs(near - 2 * far) <= 3 * max(cost)


def _rand_instance(rng, n, nb=2):
    home = [rng.randrange(nb) for _ in range(n)]
    cost = [rng.randrange(1, 50) for _ in range(n)]
    units = [rng.randrange(1, 4) for _ in range(nb)]
    return home, cost, units


@pytest.mark.parametrize("trial", range(60))
def test_load_balance_against_brute_force_minimax(trial):
    rng = random.Random(1000 + trial)
    n = rng.randrange(1, 9)
    home, cost, units = _rand_instance(rng, n)
    weighted = trial % 2 == 1
    ln, lf = (2, 3) if weighted else (1, 1)
    queues = S.cbmf_queues(home, 2)
    out = S.load_balance(queues, cost, units, ln, lf)
    assert sorted(out.queues[0] + out.queues[1]) == list(range(n))
    got = S.makespan_num_den(out.work_after, units)
    before = S.makespan_num_den(out.work_before, units)
    opt = S.brute_force_minimax(home, cost, units, ln, lf)
    # never better than the optimum, never worse than doing nothing
    assert got[0] * opt[1] >= opt[0] * got[1]
    assert got[0] * before[1] <= before[0] * got[1]
    if not weighted:
        # two banks, equal weights: makespan <= opt + (largest patch) / (all units)
        total_units = sum(units)
        lhs = got[0] * opt[1] * total_units
        rhs = opt[0] * got[1] * total_units + max(cost) * got[1] * opt[1]
        assert lhs <= rhs


def _rand_table(rng, n, nb, chunk=256):
    nch = n * 4 + 8
    m = S.BankMap(chunk, [rng.randrange(nb) for _ in range(nch)])
    patches, pos = [], 0
    for _ in range(n):
        size = rng.choice([256, 512, 768, 1024])
        patches.append((pos, pos + size))
        pos += size
    return S.bank_table(patches, [m], nb)


@pytest.mark.parametrize("trial", range(40))
def test_minimax_lpt_against_brute_force(trial):
    rng = random.Random(5000 + trial)
    n = rng.randrange(1, 8)
    t = _rand_table(rng, n, 2)
    identical = trial % 2 == 0
    units = [2, 2] if identical else [rng.randrange(1, 4), rng.randrange(1, 4)]
    ln, lf = (1, 1) if identical else (3, 4)
    queues, W = S.minimax_lpt(t, units, ln, lf)
    assert sorted(queues[0] + queues[1]) == list(range(n))
    got = S.makespan_num_den(W, units)
    opt = S.brute_force_minimax_table(t, units, ln, lf)
    assert got[0] * opt[1] >= opt[0] * got[1]            # never better than the optimum
    if identical:
        # two identical machines: Graham's LPT bound, makespan <= (4/3 - 1/6) * OPT
        assert 6 * got[0] * opt[1] <= 7 * opt[0] * got[1]


@pytest.mark.parametrize("trial", range(20))
def test_minimax_lpt_three_banks_against_brute_force(trial):
    """Three banks: every patch assigned once, never better than the exact
    optimum, and with identical units and equal weights within Graham's LPT
    bound for m = 3 machines, (4/3 - 1/9) OPT = 11/9 OPT."""
    rng = random.Random(7000 + trial)
    n = rng.randrange(1, 8)
    t = _rand_table(rng, n, 3)
    identical = trial % 2 == 0
    units = [1, 1, 1] if identical else [rng.randrange(1, 4) for _ in range(3)]
    ln, lf = (1, 1) if identical else (2, 5)
    queues, W = S.minimax_lpt(t, units, ln, lf)
    assert sorted(queues[0] + queues[1] + queues[2]) == list(range(n))
    got = S.makespan_num_den(W, units)
    opt = S.brute_force_minimax_table(t, units, ln, lf)
    assert got[0] * opt[1] >= opt[0] * got[1]
    if identical:
        assert 9 * got[0] * opt[1] <= 11 * opt[0] * got[1]


def test_minimax_queues_are_longest_first():
    m = S.BankMap(256, [0, 1] * 40)
    patches = [(0, 256), (256, 1280), (1280, 1536), (1536, 3584), (3584, 3840)]
    t = S.bank_table(patches, [m], 2)
    queues, _ = S.minimax_lpt(t, [1, 1], 1, 1)
    sizes = {i: p[1] - p[0] for i, p in enumerate(patches)}
    assert queues[0][0] == 3 and queues[1][0] == 1          # the two largest first
    for q in queues:
        assert [sizes[i] for i in q] == sorted((sizes[i] for i in q), reverse=True)
