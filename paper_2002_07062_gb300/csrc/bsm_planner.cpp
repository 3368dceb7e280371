// bsm_planner.cpp -- the scheduling steps of Sec. 4, on the host.
//
// Sec. 4.1 (Cluster Beamforming):
//   1. batch-to-bank table: for every patch, the bytes it has on every bank
//      (die), summed over the maps given (input, and output if counted), and an
//      OVERLAP flag when more than one bank holds some of it; N_b = patches with
//      any byte on bank b (sum N_b > N as soon as one patch overlaps);
//   2. every patch goes to the bank with the largest share; equal shares pick
//      one tied bank with equal probability -- here the tied bank with index
//      (splitmix64(tie_seed, patch) >> 32) mod (number tied), banks in
//      increasing order -- so that sum L_b = N;
//   3. each bank's patches form a queue, in patch order, served round robin by
//      the compute units near that bank.
// Sec. 4.2 (Load balancing, the weighted variant when l_far != l_near):
//   the most loaded bank (largest W_b / units_b, first on ties) hands its last
//   native patch to the least loaded bank (smallest, first on ties) while that
//   strictly lowers the larger of the two finish times; a moved patch costs
//   l_far per byte on its new bank, a native one l_near.  Moves are "virtual":
//   only the queue changes, the data stays where it is.
// Sec. 4.2, general form (MINIMAX: minimise the largest per-unit finish
// time; the cost of a patch depends on its distance to the unit): here the
// cost of patch i on bank b is sum_b' bytes(i, b') * (l_near if b' == b else
// l_far); patches are taken in decreasing order of their smallest cost
// (ties: lower index), each to the bank with the smallest (W_b + cost) /
// units_b (ties: lower bank) -- the longest-processing-time rule.  The
// queues keep that order, so every bank runs its longest patches first.
// All quantities are integers, so the result is exact and reproducible.

#include <algorithm>
#include <cstdint>
#include <vector>

#include "bsm_internal.h"

namespace bsm {
namespace {

uint64_t splitmix64_at(uint64_t seed, uint64_t i)
{
    uint64_t z = seed + (i + 1) * 0x9E3779B97F4A7C15ULL;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

// a / ua < b / ub, exactly
bool ratio_less(int64_t a, int64_t ua, int64_t b, int64_t ub)
{
    return static_cast<__int128>(a) * ub < static_cast<__int128>(b) * ua;
}

}  // namespace

int schedule_host(const bsm_schedule_desc *d, bsm_schedule_out *o)
{
    if (!d || !o)
        return BSM_ERR_INVALID_ARG;
    const int nb = d->n_banks;
    const int64_t np = d->n_patches;
    if (nb < 1 || nb > BSM_MAX_DIES || np < 0 || d->n_maps < 1 || d->n_maps > 2)
        return BSM_ERR_INVALID_ARG;
    if (np > INT32_MAX)
        return BSM_ERR_UNSUPPORTED;
    for (int m = 0; m < d->n_maps; ++m)
        if (d->chunk[m] <= 0 || d->n_chunks[m] < 0 || (d->n_chunks[m] > 0 && !d->bank_of_chunk[m]))
            return BSM_ERR_INVALID_ARG;
    if (np > 0 && (!d->patch_begin || !d->patch_end || !o->bytes_on_bank || !o->overlap || !o->bank ||
                   !o->queue_items || !o->moved))
        return BSM_ERR_INVALID_ARG;
    if (!o->N || !o->L || !o->queue_len)
        return BSM_ERR_INVALID_ARG;
    if (d->balance) {
        if (!d->units || (np > 0 && !d->cost) || d->l_near <= 0 || d->l_far <= 0 || !o->work_before ||
            !o->work_after)
            return BSM_ERR_INVALID_ARG;
        for (int b = 0; b < nb; ++b)
            if (d->units[b] <= 0)
                return BSM_ERR_INVALID_ARG;
    }

    // ---- Sec. 4.1 step 1: the batch-to-bank table
    for (int b = 0; b < nb; ++b)
        o->N[b] = 0;
    for (int64_t i = 0; i < np; ++i) {
        int64_t *row = o->bytes_on_bank + i * nb;
        std::fill(row, row + nb, 0);
        const int64_t lo = d->patch_begin[i], hi = d->patch_end[i];
        if (lo < 0 || hi < lo)
            return BSM_ERR_INVALID_ARG;
        for (int m = 0; m < d->n_maps; ++m) {
            const int64_t g = d->chunk[m];
            if (hi > lo && (hi - 1) / g >= d->n_chunks[m])
                return BSM_ERR_INVALID_ARG;
            for (int64_t k = lo / g; k * g < hi; ++k) {
                const int bank = d->bank_of_chunk[m][k];
                if (bank < 0 || bank >= nb)
                    return BSM_ERR_INVALID_ARG;
                const int64_t a = std::max(lo, k * g), e = std::min(hi, (k + 1) * g);
                row[bank] += e - a;
            }
        }
        int present = 0;
        for (int b = 0; b < nb; ++b)
            if (row[b] > 0) {
                ++present;
                ++o->N[b];
            }
        o->overlap[i] = present > 1 ? 1 : 0;
    }

    // ---- Sec. 4.1 step 2: resolve overlaps (majority, seeded fair tie break)
    for (int b = 0; b < nb; ++b)
        o->L[b] = 0;
    for (int64_t i = 0; i < np; ++i) {
        const int64_t *row = o->bytes_on_bank + i * nb;
        const int64_t top = *std::max_element(row, row + nb);
        int tied[BSM_MAX_DIES], nt = 0;
        for (int b = 0; b < nb; ++b)
            if (row[b] == top)
                tied[nt++] = b;
        int pick = tied[0];
        if (nt > 1)
            pick = tied[(splitmix64_at(d->tie_seed, static_cast<uint64_t>(i)) >> 32) %
                        static_cast<uint64_t>(nt)];
        o->bank[i] = pick;
        ++o->L[pick];
    }

    // ---- Sec. 4.1 step 3: per-bank queues in patch order
    std::vector<std::vector<int32_t>> q(nb);
    for (int64_t i = 0; i < np; ++i)
        q[o->bank[i]].push_back(static_cast<int32_t>(i));

    // ---- Sec. 4.2: load balance
    o->n_moved = 0;
    if (d->balance) {
        std::vector<int64_t> W(nb, 0);
        std::vector<size_t> natives(nb);   // q[b][0 .. natives[b]) are b's own patches
        for (int b = 0; b < nb; ++b) {
            for (int32_t i : q[b])
                W[b] += d->cost[i] * d->l_near;
            natives[b] = q[b].size();
            o->work_before[b] = W[b];
        }
        for (;;) {
            int a = 0, lo = 0;
            for (int b = 1; b < nb; ++b) {
                if (ratio_less(W[a], d->units[a], W[b], d->units[b]))
                    a = b;
                if (ratio_less(W[b], d->units[b], W[lo], d->units[lo]))
                    lo = b;
            }
            if (a == lo || natives[a] == 0)
                break;
            const int32_t i = q[a][natives[a] - 1];
            const int64_t wa = W[a] - d->cost[i] * d->l_near;
            const int64_t wl = W[lo] + d->cost[i] * d->l_far;
            const bool a_is_max = !ratio_less(wa, d->units[a], wl, d->units[lo]);
            const bool better = a_is_max ? ratio_less(wa, d->units[a], W[a], d->units[a])
                                         : ratio_less(wl, d->units[lo], W[a], d->units[a]);
            if (!better)
                break;
            q[a].erase(q[a].begin() + static_cast<std::ptrdiff_t>(natives[a] - 1));
            --natives[a];
            q[lo].push_back(i);
            o->moved[o->n_moved++] = i;
            W[a] = wa;
            W[lo] = wl;
        }
        for (int b = 0; b < nb; ++b)
            o->work_after[b] = W[b];
    }

    if (d->method == 1) {
        // MINIMAX by longest patch first (replaces the queues built above)
        if (!d->units || d->l_near <= 0 || d->l_far <= 0 || !o->work_after)
            return BSM_ERR_INVALID_ARG;
        for (int b = 0; b < nb; ++b)
            if (d->units[b] <= 0)
                return BSM_ERR_INVALID_ARG;
        auto cost = [&](int64_t i, int b) {
            const int64_t *row = o->bytes_on_bank + i * nb;
            int64_t c = 0;
            for (int bb = 0; bb < nb; ++bb)
                c += row[bb] * (bb == b ? d->l_near : d->l_far);
            return c;
        };
        std::vector<int64_t> key(static_cast<size_t>(np));
        std::vector<int32_t> order(static_cast<size_t>(np));
        for (int64_t i = 0; i < np; ++i) {
            int64_t mn = cost(i, 0);
            for (int b = 1; b < nb; ++b)
                mn = std::min(mn, cost(i, b));
            key[i] = mn;
            order[i] = static_cast<int32_t>(i);
        }
        std::stable_sort(order.begin(), order.end(),
                         [&](int32_t u, int32_t v) { return key[u] > key[v]; });
        std::vector<int64_t> W(nb, 0);
        for (int b = 0; b < nb; ++b)
            q[b].clear();
        for (int32_t i : order) {
            int best = 0;
            for (int b = 1; b < nb; ++b)
                if (ratio_less(W[b] + cost(i, b), d->units[b], W[best] + cost(i, best), d->units[best]))
                    best = b;
            W[best] += cost(i, best);
            q[best].push_back(i);
        }
        for (int b = 0; b < nb; ++b) {
            o->work_after[b] = W[b];
            if (o->work_before)
                o->work_before[b] = 0;
        }
    }

    int64_t pos = 0;
    for (int b = 0; b < nb; ++b) {
        o->queue_len[b] = static_cast<int64_t>(q[b].size());
        for (int32_t i : q[b])
            o->queue_items[pos++] = i;
    }
    return BSM_OK;
}

}  // namespace bsm
