"""Host planner of libbsm (C++) against the scheduling oracle (Python), on
synthetic address maps: the Sec. 4.1 table, overlap resolution and the
Sec. 4.2 load balance must agree exactly (integer results)."""
import json
import os
import random

import pytest

from oracle import schedule_oracle as S
from paper_2002_07062_gb300 import bsm

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()


def _oracle(patches, maps, nb, seed, balance, units, ln, lf, cost):
    t = S.bank_table(patches, [S.BankMap(c, b) for c, b in maps], nb)
    bank = S.resolve_overlap(t, seed)
    out = {"bytes_on_bank": t.bytes_on_bank, "overlap": t.overlap, "N": t.N, "bank": bank,
           "L": S.counts(bank, nb)}
    q = S.cbmf_queues(bank, nb)
    if balance:
        r = S.load_balance(q, cost, units, ln, lf)
        out.update(queues=r.queues, moved=r.moved, work_before=r.work_before,
                   work_after=r.work_after)
    else:
        out.update(queues=q, moved=[])
    return out


def _compare(got, want, balance):
    for k in ("bytes_on_bank", "overlap", "N", "bank", "L", "queues", "moved"):
        assert got[k] == want[k], k
    if balance:
        assert got["work_before"] == want["work_before"]
        assert got["work_after"] == want["work_after"]


def test_paper_table_fixture():
    g = json.load(open(os.path.join(GOLDEN, "batch_bank_table.json")))
    patches = [tuple(p) for p in g["patches"]]
    got = bsm.bsm_schedule_host(patches, [(g["chunk"], g["bank_of_chunk"])], 4, 1)
    assert [[1 if v else 0 for v in row] for row in got["bytes_on_bank"]] == g["table"]
    assert got["overlap"] == g["overlap"] and got["N"] == g["N"]
    assert got["bank"] == g["resolved_bank"] and got["L"] == g["L"]


@pytest.mark.parametrize("trial", range(40))
def test_random_instances_match_oracle(trial):
    rng = random.Random(trial)
    nb = rng.choice([2, 2, 3, 4])
    chunk = rng.choice([128, 256, 4096])
    n = rng.randrange(0, 120)
    sizes = [rng.choice([128, 256, 384, 1024, 4096, 5000]) for _ in range(n)]
    patches, pos = [], 0
    for s in sizes:
        patches.append((pos, pos + s))
        pos += s + rng.choice([0, 0, 16, 128])
    nch = pos // chunk + 1
    kind = rng.choice(["random", "runs", "one_bank", "alternate"])
    if kind == "random":
        m = [rng.randrange(nb) for _ in range(nch)]
    elif kind == "runs":
        m, b = [], 0
        while len(m) < nch:
            m += [b] * rng.randrange(1, 9)
            b = rng.randrange(nb)
        m = m[:nch]
    elif kind == "one_bank":
        m = [0] * nch
    else:
        m = [k % nb for k in range(nch)]
    maps = [(chunk, m)]
    if rng.random() < 0.5:
        maps.append((chunk, [rng.randrange(nb) for _ in range(nch)]))
    seed = rng.getrandbits(64)
    balance = rng.random() < 0.7
    units = [rng.randrange(1, 80) for _ in range(nb)]
    ln = rng.randrange(1, 600)
    lf = ln + rng.randrange(0, 400)
    cost = [2 * (e - b) for b, e in patches]
    got = bsm.bsm_schedule_host(patches, maps, nb, seed, balance, units, ln, lf, cost)
    want = _oracle(patches, maps, nb, seed, balance, units, ln, lf, cost)
    _compare(got, want, balance)


def test_degenerate_first_portion_map_balances():
    n = 200
    patches = [(k * 4096, (k + 1) * 4096) for k in range(n)]
    maps = [(4096, [0] * n)]
    got = bsm.bsm_schedule_host(patches, maps, 2, 0, True, [76, 76], 1, 1, [8192] * n)
    assert got["L"] == [n, 0]
    assert [len(q) for q in got["queues"]] == [100, 100]
    want = _oracle(patches, maps, 2, 0, True, [76, 76], 1, 1, [8192] * n)
    _compare(got, want, True)


@pytest.mark.parametrize("trial", range(30))
def test_minimax_matches_oracle(trial):
    rng = random.Random(900 + trial)
    nb = rng.choice([2, 2, 3])
    chunk = rng.choice([128, 1024])
    n = rng.randrange(0, 200)
    sizes = [rng.choice([256, 1024, 4096, 32768, 8192]) for _ in range(n)]
    patches, pos = [], 0
    for sz in sizes:
        patches.append((pos, pos + sz))
        pos += sz
    nch = pos // chunk + 1
    maps = [(chunk, [rng.randrange(nb) for _ in range(nch)])]
    units = [rng.randrange(1, 80) for _ in range(nb)]
    ln = rng.randrange(1, 500)
    lf = ln + rng.randrange(0, 300)
    got = bsm.bsm_schedule_host(patches, maps, nb, 0, False, units, ln, lf, minimax=True)
    t = S.bank_table(patches, [S.BankMap(c, b) for c, b in maps], nb)
    queues, W = S.minimax_lpt(t, units, ln, lf)
    assert got["queues"] == queues
    assert got["work_after"] == W
