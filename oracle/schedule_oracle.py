"""schedule_oracle.py -- TEST INFRASTRUCTURE ONLY.

Plain-Python restatement of the paper's two scheduling steps, written from the
text of Sec. 4 of "An optimal scheduling architecture for accelerating batch
algorithms on Neural Network processor architectures" (Nyshadham et al.):

* Sec. 4.1, Cluster Beamforming (CBMF): build the batch-to-bank table (for
  every patch, which memory banks hold its bytes, with an OVERLAP flag), count
  N_b patches per bank (the sum exceeds N when patches overlap), resolve every
  overlapping patch to the bank holding the largest share (equal shares: each
  tied bank with equal probability), which gives L_b with sum L_b = N; then
  the patches of each bank are handed, round robin, to the compute units near
  that bank.
* Sec. 4.2, Load balancing (LB): move patches from over-loaded banks to
  under-loaded ones ("virtual" assignment: the data is not moved), optionally
  weighted so that far units take load in inverse proportion to latency; the
  MINIMAX objective of Sec. 4.2 (minimise the largest per-unit execution time)
  is the quantity the move rule must never worsen.

The figures that would fix the details (Fig-1, Fig-2) are missing from the
paper text, so the readings below are this project's:

* bytes of a patch on a bank = bytes of its input range plus (optionally) its
  output range that the address map places on that bank;
* the equal-probability tie break is a fair choice driven by splitmix64
  (Steele, Lea and Flood 2014, with the constants Vigna published) on
  (tie_seed, patch index), so plans are reproducible;
* the load-balance move rule: the most loaded bank gives its last native
  patch to the least loaded bank while that strictly lowers the larger of the
  two banks' estimated finish times; finish time of bank b =
  (sum of native patch bytes * l_near + sum of moved-in patch bytes * l_far)
  / (compute units on b); everything is integer, so any faithful
  implementation reproduces it exactly.

This module is independent of the CUDA library: it imports nothing from the
package and is imported only by tests and by bench.py's CPU leg.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from itertools import product
from typing import List, Optional, Sequence, Tuple

MASK64 = (1 << 64) - 1
GOLDEN_GAMMA = 0x9E3779B97F4A7C15


def splitmix64(seed: int, i: int) -> int:
    """Output number i (0-based) of a splitmix64 generator whose state starts at
    `seed`: the state advances by the golden gamma, then is mixed."""
    z = (seed + (i + 1) * GOLDEN_GAMMA) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


@dataclass
class BankMap:
    """Bank (die) of every `chunk`-byte chunk of one buffer, chunk k covering
    bytes [k*chunk, (k+1)*chunk)."""
    chunk: int
    bank_of_chunk: Sequence[int]


@dataclass
class BankTable:
    """The Sec. 4.1 batch-to-bank table."""
    bytes_on_bank: List[List[int]]  # [patch][bank]
    overlap: List[int]              # 1 when the patch lies on more than one bank
    N: List[int]                    # patches with any byte on bank b


def _bytes_per_bank(lo: int, hi: int, m: BankMap, n_banks: int) -> List[int]:
    out = [0] * n_banks
    pos = lo
    while pos < hi:
        k = pos // m.chunk
        end = min(hi, (k + 1) * m.chunk)
        out[m.bank_of_chunk[k]] += end - pos
        pos = end
    return out


def bank_table(patches: Sequence[Tuple[int, int]], maps: Sequence[BankMap],
               n_banks: int) -> BankTable:
    """patches[i] = (first byte, one past last byte) of patch i; the same byte
    range is looked up in every map in `maps` (the input buffer, and the output
    buffer when its bytes count too) and the bytes are added."""
    table, overlap = [], []
    for lo, hi in patches:
        row = [0] * n_banks
        for m in maps:
            for b, v in enumerate(_bytes_per_bank(lo, hi, m, n_banks)):
                row[b] += v
        table.append(row)
        overlap.append(1 if sum(1 for v in row if v > 0) > 1 else 0)
    N = [sum(1 for row in table if row[b] > 0) for b in range(n_banks)]
    return BankTable(table, overlap, N)


def resolve_overlap(table: BankTable, tie_seed: int) -> List[int]:
    """Bank of every patch: the bank with the largest share; equal shares pick
    one of the tied banks (in increasing bank order) with index
    (splitmix64(tie_seed, patch) >> 32) mod (number tied)."""
    bank = []
    for i, row in enumerate(table.bytes_on_bank):
        top = max(row)
        tied = [b for b, v in enumerate(row) if v == top]
        if len(tied) == 1:
            bank.append(tied[0])
        else:
            bank.append(tied[(splitmix64(tie_seed, i) >> 32) % len(tied)])
    return bank


def counts(bank: Sequence[int], n_banks: int) -> List[int]:
    """L_b, the number of patches assigned to bank b."""
    return [sum(1 for b in bank if b == k) for k in range(n_banks)]


def cbmf_queues(bank: Sequence[int], n_banks: int) -> List[List[int]]:
    """Per-bank queue in patch order; the near units of a bank take its
    patches round robin in this order."""
    return [[i for i, b in enumerate(bank) if b == k] for k in range(n_banks)]


@dataclass
class Balanced:
    queues: List[List[int]]
    moved: List[int] = field(default_factory=list)   # patch ids in move order
    work_before: List[int] = field(default_factory=list)
    work_after: List[int] = field(default_factory=list)


def _finish_less(wa: int, na: int, wb: int, nb: int) -> bool:
    """wa/na < wb/nb without division."""
    return wa * nb < wb * na


def load_balance(queues: Sequence[Sequence[int]], cost: Sequence[int],
                 units: Sequence[int], l_near: int, l_far: int) -> Balanced:
    """Sec. 4.2 load balancing on per-bank queues.

    cost[i]  -- work of patch i (bytes it moves);
    units[b] -- compute units near bank b;
    l_near, l_far -- latency of a near / far access (equal values give the
                     unweighted variant).
    Work of bank b: W_b = l_near * (native bytes) + l_far * (moved-in bytes);
    its finish time is W_b / units[b].
    """
    nb = len(queues)
    q = [list(x) for x in queues]
    W = [sum(cost[i] for i in lst) * l_near for lst in q]
    before = list(W)
    moved: List[int] = []
    native = [list(lst) for lst in q]          # natives still on their home bank
    while True:
        a = 0
        for b in range(1, nb):
            if _finish_less(W[a], units[a], W[b], units[b]):
                a = b
        lo = 0
        for b in range(1, nb):
            if _finish_less(W[b], units[b], W[lo], units[lo]):
                lo = b
        if a == lo or not native[a]:
            break
        i = native[a][-1]
        wa = W[a] - cost[i] * l_near
        wl = W[lo] + cost[i] * l_far
        # accept only if max(wa/ua, wl/ul) < W[a]/ua
        new_max_a = not _finish_less(wa, units[a], wl, units[lo])   # wa/ua >= wl/ul
        if new_max_a:
            better = _finish_less(wa, units[a], W[a], units[a])
        else:
            better = _finish_less(wl, units[lo], W[a], units[a])
        if not better:
            break
        native[a].pop()
        q[a].remove(i)
        q[lo].append(i)
        moved.append(i)
        W[a], W[lo] = wa, wl
    return Balanced(q, moved, before, W)


def makespan_num_den(W: Sequence[int], units: Sequence[int]) -> Tuple[int, int]:
    """max_b W_b / units[b] as an exact fraction (numerator, denominator)."""
    best = (W[0], units[0])
    for b in range(1, len(W)):
        if _finish_less(best[0], best[1], W[b], units[b]):
            best = (W[b], units[b])
    return best


def brute_force_minimax(home: Sequence[int], cost: Sequence[int], units: Sequence[int],
                        l_near: int, l_far: int) -> Tuple[int, int]:
    """Exact optimum of the Sec. 4.2 MINIMAX problem on a tiny instance, with
    the cost of patch i on bank b = cost[i] * (l_near if b is its home else
    l_far); returns the optimal largest finish time as a fraction."""
    nb = len(units)
    best: Optional[Tuple[int, int]] = None
    for assign in product(range(nb), repeat=len(cost)):
        W = [0] * nb
        for i, b in enumerate(assign):
            W[b] += cost[i] * (l_near if b == home[i] else l_far)
        ms = makespan_num_den(W, units)
        if best is None or _finish_less(ms[0], ms[1], best[0], best[1]):
            best = ms
    assert best is not None
    return best


def minimax_lpt(table: BankTable, units: Sequence[int], l_near: int, l_far: int):
    """Sec. 4.2 MINIMAX (minimise the largest per-unit finish time) by the
    longest-processing-time rule: the cost of patch i on bank b is
    sum over banks b' of bytes_on_bank[i][b'] * (l_near if b' == b else
    l_far); patches go in decreasing order of their smallest cost (ties:
    lower index first), each to the bank whose finish time after taking it,
    (W_b + cost) / units[b], is smallest (ties: lower bank).  Returns the
    per-bank queues in assignment order and the final W."""
    nb = len(units)
    rows = table.bytes_on_bank

    def cost(i, b):
        return sum(v * (l_near if bb == b else l_far) for bb, v in enumerate(rows[i]))

    order = sorted(range(len(rows)), key=lambda i: (-min(cost(i, b) for b in range(nb)), i))
    W = [0] * nb
    queues: List[List[int]] = [[] for _ in range(nb)]
    for i in order:
        best = 0
        for b in range(1, nb):
            # (W_b + c_b) / u_b < (W_best + c_best) / u_best
            if _finish_less(W[b] + cost(i, b), units[b], W[best] + cost(i, best), units[best]):
                best = b
        W[best] += cost(i, best)
        queues[best].append(i)
    return queues, W


def brute_force_minimax_table(table: BankTable, units: Sequence[int], l_near: int,
                              l_far: int) -> Tuple[int, int]:
    """Exact optimum of the same problem (every assignment tried)."""
    nb = len(units)
    rows = table.bytes_on_bank
    best: Optional[Tuple[int, int]] = None
    for assign in product(range(nb), repeat=len(rows)):
        W = [0] * nb
        for i, b in enumerate(assign):
            W[b] += sum(v * (l_near if bb == b else l_far) for bb, v in enumerate(rows[i]))
        ms = makespan_num_den(W, units)
        if best is None or _finish_less(ms[0], ms[1], best[0], best[1]):
            best = ms
    assert best is not None
    return best
