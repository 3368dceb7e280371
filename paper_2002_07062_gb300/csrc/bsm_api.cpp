// bsm_api.cpp -- the C ABI of libbsm (include/bsm.h): argument checks, plan
// construction (patches, die queues, upload of the patch table -- the
// "Patch<->Cluster mapping table" kept in device memory, Sec. 5), plan
// execution, the plan cache behind the one-call entry points, and status.

#include <cuda_runtime.h>

#include <algorithm>
#include <atomic>
#include <chrono>
#include <cmath>
#include <cstddef>
#include <cstring>
#include <list>
#include <mutex>
#include <new>
#include <numeric>
#include <string>
#include <vector>

#include "bsm_internal.h"
#include "bsm_trace.h"

namespace bsm {

namespace {
thread_local std::string t_last_error;
}

int record_cuda_error(int cuda_error, const char *where)
{
    const cudaError_t e = static_cast<cudaError_t>(cuda_error);
    t_last_error = std::string(where) + ": " + cudaGetErrorName(e) + " (" + cudaGetErrorString(e) + ")";
    return BSM_ERR_CUDA;
}

int topology_get(int device, int force, bsm_topology *out);
int die_check_host(int device, const void *ptr, int64_t bytes, int64_t chunk, const int8_t *die_of_chunk,
                   const int8_t *sm_group, int invert, uint32_t *xor_out, float *ms_out);
int probe_latency_host(int device, const std::vector<int64_t> &lines, int reps, std::vector<float> &lat,
                       std::vector<int32_t> &seen);

namespace {

constexpr int kMaxDevices = 64;
constexpr uint64_t kDefaultTieSeed = 0x2002070600ull;
constexpr int64_t kMaxMapChunks = 1ll << 24;

struct DeviceCtx {
    bool ready = false;
    int n_sm = 0;
    int smem_optin = 0;
    uint32_t *status = nullptr;   // sticky device status word
};

std::mutex g_mu;
DeviceCtx g_dev[kMaxDevices];
std::atomic<int> g_checked{0};

int cuda_error(cudaError_t e, const char *where) { return record_cuda_error(static_cast<int>(e), where); }

int device_ctx(int device, DeviceCtx **out)
{
    if (device < 0) {
        if (cudaGetDevice(&device) != cudaSuccess)
            return BSM_ERR_NO_DEVICE;
    }
    if (device >= kMaxDevices)
        return BSM_ERR_NO_DEVICE;
    std::lock_guard<std::mutex> lk(g_mu);
    DeviceCtx &c = g_dev[device];
    if (!c.ready) {
        int prev = -1;
        cudaGetDevice(&prev);
        if (cudaSetDevice(device) != cudaSuccess)
            return BSM_ERR_NO_DEVICE;
        int rc = BSM_OK;
        if (cudaDeviceGetAttribute(&c.n_sm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
            cudaDeviceGetAttribute(&c.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, device) !=
                cudaSuccess)
            rc = BSM_ERR_NO_DEVICE;
        cudaError_t e = cudaSuccess;
        if (!rc && (e = static_cast<cudaError_t>(kernel_set_smem_limit(c.smem_optin))) != cudaSuccess)
            rc = cuda_error(e, "cudaFuncSetAttribute");
        if (!rc && (e = cudaMalloc(&c.status, 256)) != cudaSuccess)
            rc = cuda_error(e, "cudaMalloc(status)");
        if (!rc && (e = cudaMemset(c.status, 0, 256)) != cudaSuccess)
            rc = cuda_error(e, "cudaMemset(status)");
        if (!rc && (e = cudaDeviceSynchronize()) != cudaSuccess)
            rc = cuda_error(e, "cudaDeviceSynchronize");
        if (prev >= 0 && prev != device)
            cudaSetDevice(prev);
        if (rc) {
            if (c.status)
                cudaFree(c.status);
            c.status = nullptr;
            return rc;
        }
        c.ready = true;
    }
    *out = &c;
    return BSM_OK;
}

}  // namespace

// The sticky status word of a device, shared by every kernel of the library.
int device_status_word(int device, uint32_t **out)
{
    DeviceCtx *c = nullptr;
    if (int rc = device_ctx(device, &c))
        return rc;
    *out = c->status;
    return BSM_OK;
}

namespace {

int64_t max_row_bytes_for(int64_t smem_optin)
{
    return ((smem_optin - kSmemHeader) / 2) & ~int64_t(127);
}

int64_t max_row_bytes_for(const DeviceCtx &c) { return max_row_bytes_for(static_cast<int64_t>(c.smem_optin)); }

int esize(int dtype) { return dtype == BSM_F32 ? 4 : 2; }

}  // namespace
}  // namespace bsm

struct bsm_plan {
    int device = 0;
    int policy = 0;
    int dtype = 0;
    int op = 0;          // BSM_OP_* of the plan
    int kernel_op = 0;   // the kernel instance it launches (bsm::Op)
    bsm::KernelArgs args{};
    int grid = 0;
    struct Launch {
        int32_t begin, end, grid, phase;
    };
    bsm::KernelArgs args1{};         // phase 1 of plans with rows longer than a stage
    int64_t n_phase1 = 0;
    bsm::KernelArgs argsg{};         // rows over groups of CTAs (one cooperative launch)
    int64_t n_group = 0;
    int grid_g = 0;
    std::vector<Launch> whole_gpu;   // WHOLE_GPU: one launch per slice
    cudaGraphExec_t whole_graph = nullptr;   // ... captured once as a CUDA graph (or null)
    void *blob = nullptr;            // device tables (patches, slice index, sm_die, heads)
    bsm_plan_stats stats{};
    // the schedule as built (bsm_plan_get_schedule): the phase-0 patch index
    // (slice order) of every queue slot, the address -> die maps and the
    // planner's inputs
    std::vector<int32_t> queue;
    int32_t q_begin[BSM_MAX_DIES] = {0, 0, 0, 0}, q_len[BSM_MAX_DIES] = {0, 0, 0, 0};
    int32_t q_count = 0;
    std::vector<int8_t> xmap, ymap;
    std::vector<int32_t> moved;
    int64_t map_chunk = 0;
    int32_t units[BSM_MAX_DIES] = {0, 0, 0, 0};
    int64_t w_near = 0, w_far = 0;
    int count_y = 0;
    uint64_t tie_seed = 0;
    // identity of the plan for the cache
    const void *x = nullptr;
    void *y = nullptr;
    uint32_t flags = 0;
    std::vector<int64_t> key_offsets;
    std::vector<int32_t> key_rows, key_cols;
    int64_t key_B = -1, key_R = -1, key_C = -1;
};

namespace bsm {
namespace {

struct SliceView {
    int64_t off;
    int32_t R, C;
};

// Validate a descriptor; fills the slice list and the element extent.
int validate(const bsm_plan_desc *d, std::vector<SliceView> &slices,
             int64_t &total_elems, int64_t &max_row_bytes)
{
    if (d->dtype != BSM_F32 && d->dtype != BSM_BF16)
        return BSM_ERR_INVALID_ARG;
    if (d->policy < BSM_POLICY_WHOLE_GPU || d->policy > BSM_POLICY_MINIMAX)
        return BSM_ERR_INVALID_ARG;
    if (d->flags & ~BSM_FLAG_CAUSAL)
        return BSM_ERR_INVALID_ARG;
    if (d->op != BSM_OP_FORWARD && d->op != BSM_OP_BACKWARD)
        return BSM_ERR_INVALID_ARG;
    if (d->op == BSM_OP_BACKWARD && d->flags)
        return BSM_ERR_INVALID_ARG;
    if (d->num_slices < 0 || d->rows_per_item < 0)
        return BSM_ERR_INVALID_ARG;
    if (d->num_slices > 0 && (!d->rows || !d->cols))
        return BSM_ERR_INVALID_ARG;
    const int es = esize(d->dtype);
    slices.clear();
    slices.reserve(static_cast<size_t>(d->num_slices));
    total_elems = 0;
    max_row_bytes = 0;
    int64_t packed = 0;
    bool misaligned = false;
    for (int64_t s = 0; s < d->num_slices; ++s) {
        const int64_t R = d->rows[s], C = d->cols[s];
        if (R < 0 || C < 1)
            return BSM_ERR_INVALID_ARG;
        const int64_t off = d->offsets ? d->offsets[s] : packed;
        if (off < 0)
            return BSM_ERR_INVALID_ARG;
        if (R > 0 && C > (int64_t(1) << 40) / R)
            return BSM_ERR_INVALID_ARG;
        const int64_t n = R * C;
        if (off > (int64_t(1) << 61) - n)
            return BSM_ERR_INVALID_ARG;
        packed = off + n;
        if (R > 0) {
            if ((C * es) % 16 != 0 || (off * es) % 16 != 0)
                misaligned = true;
            max_row_bytes = std::max(max_row_bytes, C * es);
            total_elems = std::max(total_elems, off + n);
        }
        slices.push_back({off, static_cast<int32_t>(R), static_cast<int32_t>(C)});
    }
    if (total_elems > 0) {
        if (!d->x || !d->y)
            return BSM_ERR_INVALID_ARG;
        const uintptr_t xa = reinterpret_cast<uintptr_t>(d->x), ya = reinterpret_cast<uintptr_t>(d->y);
        const uintptr_t len = static_cast<uintptr_t>(total_elems) * es;
        if (xa != ya && xa < ya + len && ya < xa + len)
            return BSM_ERR_INVALID_ARG;   // partial overlap
        if ((xa & 15) || (ya & 15))
            misaligned = true;
        if (d->op == BSM_OP_BACKWARD) {
            if (!d->x2)
                return BSM_ERR_INVALID_ARG;
            const uintptr_t ga = reinterpret_cast<uintptr_t>(d->x2);
            if (ga != ya && ga < ya + len && ya < ga + len)
                return BSM_ERR_INVALID_ARG;
            if (ga & 15)
                misaligned = true;
        }
    }
    if (misaligned)
        return BSM_ERR_MISALIGNED;
    // slices must not overlap one another
    if (d->offsets && slices.size() > 1) {
        std::vector<size_t> order;
        order.reserve(slices.size());
        for (size_t s = 0; s < slices.size(); ++s)
            if (slices[s].R > 0)
                order.push_back(s);
        std::sort(order.begin(), order.end(),
                  [&](size_t a, size_t b) { return slices[a].off < slices[b].off; });
        for (size_t k = 1; k < order.size(); ++k) {
            const SliceView &p = slices[order[k - 1]];
            if (p.off + int64_t(p.R) * p.C > slices[order[k]].off)
                return BSM_ERR_INVALID_ARG;
        }
    }
    return BSM_OK;
}

// The patch table of a plan: a host computation from the descriptor and two
// figures of the device (its SM count and the opt-in shared memory of a
// block), with no CUDA call.
struct PatchLayout {
    int64_t stage = 0;                  // bytes per shared-memory stage
    int n_stages = 0;
    std::vector<Item> items;            // phase 0, in slice order
    std::vector<LongSeg> segs;          // parallel to items when there are long rows
    std::vector<Item> items1;           // phase 1: the segments of rows cut into several
    std::vector<LongSeg> segs1;
    std::vector<int32_t> slice_first, slice_first1;
    int64_t n_parts = 0;                // segments of rows cut into several
    int64_t long_rows = 0;              // rows longer than a stage
    // rows split over groups of CTAs (forward): one record per row, slice
    // order; the group launch's own stage figures
    std::vector<Item> items_g;
    std::vector<int32_t> slice_first_g;
    int32_t group_k = 0, n_groups = 0;
    int64_t stage_g = 0;
    int n_stages_g = 0;
};

// Rows over groups of CTAs (forward pass).  A row longer than one stage is
// cut into K parts, each staged by one CTA of a group of K (one read of every
// element, one launch).  K: the fewest CTAs whose parts fit the consumer
// threads' registers (64 KiB) and a third of the shared memory (groups of
// n_sm / K CTAs; n_sm mod K SMs stay idle).  Used for rows of at least
// kGroupMinParts parts on groups of at most kGroupMaxSize CTAs, when the
// batch's long rows fill the groups' waves at least two thirds (so the one
// launch beats the two-launch cut of few long rows into segments, which
// reads each row twice); K depends on the longest such row and the device
// only, never on the policy.
constexpr int64_t kGroupMinParts = 5;    // rows of fewer parts stay on one CTA
constexpr int64_t kGroupMaxSize = 32;    // larger groups wait too long on their slowest member

int choose_groups(const std::vector<SliceView> &slices, int es, int n_sm, int64_t smem_optin, PatchLayout &L)
{
    const int64_t avail = smem_optin - kSmemHeader;
    const int64_t long_cap = max_row_bytes_for(smem_optin);
    const int64_t vec = 16 / es;                 // elements per 16-byte vector
    int64_t n_cand = 0, lmax = 0;
    for (const SliceView &v : slices)
        if (v.R > 0 && int64_t(v.C) * es > long_cap) {
            n_cand += v.R;
            lmax = std::max<int64_t>(lmax, v.C);
        }
    if (n_cand == 0)
        return 0;
    auto stage_for = [&](int64_t k) {
        const int64_t part = ((lmax + k - 1) / k + vec - 1) / vec * vec;
        return (part * es + 127) & ~int64_t(127);
    };
    // a part fits a third of the shared memory (three stages) and the
    // registers of the consumer threads (kGroupVecs vectors each)
    const int64_t part_cap = std::min<int64_t>((avail / 3) & ~int64_t(127),
                                               int64_t(kGroupVecs) * 16 * kConsumerWarps * 32);
    const int64_t kmin = std::max<int64_t>(2, (lmax * es + part_cap - 1) / part_cap);
    // The smallest group whose parts fit: a member's time per row goes by
    // the vectors each of its threads holds (kGroupVecs at the cap), so the
    // fewest members with full parts move the most bytes per exchange, even
    // when n_sm / K groups leave SMs idle.  Measured on GB300 (256 MiB of
    // rows, GB/s): fp32 1 MiB rows K = 16 (9 groups) 4746 against K = 19 (8
    // groups) 4347, 17 and 18 lower still; bf16 1 MiB the same (3952 against
    // 3635); bf16 512 KiB K = 8 4139 against K = 16 2612 and K = 19 2316;
    // fp32 2 MiB K = 32 4336 against K = 38 3748.  Against the paths that
    // stream a row twice through one CTA: groups of 2 and 4 lose (bf16
    // 128 KiB 4006 against 4500, fp32 256 KiB 4709 against 4886), whose
    // second read mostly hits L2 and which wait on no other CTA; groups of
    // 64 lose to the two-launch segments (fp32 4 MiB rows 3612 against
    // 3983), while fp32 2 MiB rows gain at K = 32 (4318 against 3978).  bf16
    // rows of 1.75 and 2 MiB (K = 28, 32) lost a little to the segments with
    // scalar arithmetic in the group routines (3570 against 3602) and gain
    // with pair arithmetic (4042 against 3700, 3756 against 3650).
    int64_t best_k = 0;
    for (int64_t k = kmin; k <= std::min<int64_t>(int64_t(kMaxGroup), int64_t(n_sm)); ++k)
        if (avail / stage_for(k) >= 3 && stage_for(k) <= part_cap) {
            best_k = k;
            break;
        }
    if (best_k == 0 || kmin < kGroupMinParts || best_k > kGroupMaxSize)
        return 0;
    const int64_t G = n_sm / best_k;
    const int64_t waves = (n_cand + G - 1) / G;
    if (3 * n_cand < 2 * waves * G)
        return 0;
    L.group_k = static_cast<int32_t>(best_k);
    L.n_groups = static_cast<int32_t>(G);
    L.stage_g = stage_for(best_k);
    L.n_stages_g = static_cast<int>(std::min<int64_t>(kMaxStages, avail / L.stage_g));
    return 1;
}

int cut_patches(const bsm_plan_desc *d, const std::vector<SliceView> &slices, int64_t max_row, int n_sm,
                int64_t smem_optin, PatchLayout &L)
{
    const int es = esize(d->dtype);
    // ---- rows over groups of CTAs first; the other rows set the stages
    const bool groups = d->op == BSM_OP_FORWARD && choose_groups(slices, es, n_sm, smem_optin, L);
    const int64_t long_cap = max_row_bytes_for(smem_optin);
    auto is_group_row = [&](const SliceView &v) { return groups && v.R > 0 && int64_t(v.C) * es > long_cap; };
    if (groups) {
        max_row = 0;
        for (const SliceView &v : slices)
            if (v.R > 0 && !is_group_row(v))
                max_row = std::max<int64_t>(max_row, int64_t(v.C) * es);
    }
    // ---- stages: one CTA per SM, as many stages as fit the shared memory
    const int64_t avail = smem_optin - kSmemHeader;
    const int in_arrays = d->op == BSM_OP_BACKWARD ? 2 : 1;   // inputs sharing a stage
    // a stage holds the longest row (for the backward pass: the row of y and
    // the row of dy), up to half the shared memory; longer rows go through
    // the stages in chunks, twice
    const int64_t row_cap = std::min<int64_t>((max_row + 127) & ~int64_t(127),
                                              (max_row_bytes_for(smem_optin) / in_arrays) & ~int64_t(127));
    const int64_t min_stage = kMinStageBytes;
    int64_t stage = std::max<int64_t>(min_stage, in_arrays * row_cap);
    // Rows longer than that cap but whose halves fit three stages (with the
    // shorter rows of the batch): stages of half such a row, so that each of
    // them (two chunks) stays staged for its second pass while the third
    // stage takes the next row's first chunk -- one copy per row
    if (max_row > max_row_bytes_for(smem_optin) / in_arrays) {
        int64_t max_short = 0;
        for (const SliceView &v : slices)
            if (v.R > 0 && int64_t(v.C) * es <= max_row_bytes_for(smem_optin) / in_arrays)
                max_short = std::max<int64_t>(max_short, int64_t(v.C) * es);
        const int64_t half = std::max<int64_t>((max_short + 127) & ~int64_t(127),
                                               ((max_row + 1) / 2 + 127) & ~int64_t(127));
        const int64_t two_chunk = std::max<int64_t>(min_stage, in_arrays * half);
        if (3 * two_chunk <= avail)
            stage = two_chunk;
        else if (d->op == BSM_OP_FORWARD && es == 4 && max_row > 2 * row_cap)
            // fp32 rows streamed in more than two chunks of the cap: three
            // stages of a third of the shared memory rather than two of the
            // cap, so that a chunk is on its way while one is written and one
            // computed (measured, same box: 256 KiB rows 4890 -> 5061 GB/s,
            // 4 MiB rows 3950 -> 3977; bf16 2 MiB rows lose, 3609 -> 3533, and
            // keep two stages; four stages gain nothing).  Rows of two chunks
            // of the cap keep them: the smaller stages would cut them into
            // three and re-read more (160 KiB rows 5235 against 4878)
            stage = std::min<int64_t>(stage, std::max<int64_t>(min_stage, (avail / 3) & ~int64_t(127)));
        else if (d->op == BSM_OP_BACKWARD) {
            // the backward pass's rows streamed by one CTA each (at least two
            // waves of them): three stages as well (same box: fp32 256 KiB
            // rows 5240 -> 5382 GB/s, bf16 128 KiB 5519 -> 5952, bf16 512 KiB
            // 4411 -> 4468); rows cut into segments over two launches keep
            // two (they lose 0.2-0.5 %)
            int64_t n_over = 0;
            for (const SliceView &v : slices)
                if (v.R > 0 && int64_t(v.C) * es > max_row_bytes_for(smem_optin) / in_arrays)
                    n_over += v.R;
            if (n_over >= 2 * int64_t(n_sm))
                stage = std::min<int64_t>(stage, std::max<int64_t>(min_stage, (avail / 3) & ~int64_t(255)));
        }
    }
    const int n_stages = static_cast<int>(std::min<int64_t>(kMaxStages, avail / stage));
    if (n_stages < 2)
        return BSM_ERR_UNSUPPORTED;
    L.stage = stage;
    L.n_stages = n_stages;

    // ---- patches: consecutive rows filling (at most) one stage.  Under the
    // queue policies a patch may run on into the next slices when they have
    // the same shape and follow back to back (a "segment"); under RR and
    // WHOLE_GPU a patch stays inside its slice, the unit those policies place.
    const bool spanning = d->policy == BSM_POLICY_DYNAMIC || d->policy == BSM_POLICY_CBMF ||
                          d->policy == BSM_POLICY_CBMF_LB || d->policy == BSM_POLICY_MINIMAX;
    std::vector<Item> &items = L.items;
    std::vector<int32_t> &slice_first = L.slice_first;
    slice_first.assign(slices.size() + 1, 0);
    // rows longer than a stage: when they are too few to fill two waves of
    // the SMs, cut into segments of whole chunks, about eight per SM over the
    // batch, so that a few long rows still spread over the device (two
    // launches, see LongSeg; eight rather than four evens out the last wave
    // of each launch: +1 to +6.5 % measured, sixteen is no better); otherwise
    // each row is one segment that one CTA streams twice within the launch
    // (its second read mostly hits L2)
    int64_t n_long_rows = 0, n_short_rows = 0;
    for (const SliceView &v : slices) {
        if (is_group_row(v))
            continue;
        if (v.R > 0 && int64_t(v.C) * es > stage / in_arrays)
            n_long_rows += v.R;
        else
            n_short_rows += v.R;
    }
    // Under the queue policies a CTA claims kFetch patches at a time, one at
    // a time on a short queue (fewer than 2 * kFetch patches per SM).  A
    // batch of fewer stage-filling patches than SMs (up to about 10 MB) is
    // therefore cut into about one patch per SM -- at most
    // ceil(rows / SMs) rows each -- so that every SM takes one patch with one
    // claim and one copy (8 x 64 x 64 fp32 ran on 2 SMs with whole-stage
    // patches).  RR and WHOLE_GPU keep their own units.
    const int64_t spread_rows = std::max<int64_t>(1, (n_short_rows + n_sm - 1) / n_sm);
    const int64_t chunk_elems = stage / in_arrays / es;
    const int64_t want_segs = n_long_rows > 0 && n_long_rows < 2 * n_sm
                                  ? std::max<int64_t>(1, (8 * n_sm + n_long_rows - 1) / n_long_rows)
                                  : 1;
    std::vector<LongSeg> &segs = L.segs;
    std::vector<Item> &items1 = L.items1;
    std::vector<LongSeg> &segs1 = L.segs1;
    std::vector<int32_t> &slice_first1 = L.slice_first1;
    slice_first1.assign(slices.size() + 1, 0);
    int64_t &n_parts = L.n_parts;
    int64_t &long_rows = L.long_rows;
    L.slice_first_g.assign(slices.size() + 1, 0);
    size_t s = 0;
    while (s < slices.size()) {
        slice_first[s] = static_cast<int32_t>(items.size());
        slice_first1[s] = static_cast<int32_t>(items1.size());
        L.slice_first_g[s] = static_cast<int32_t>(L.items_g.size());
        const SliceView &v = slices[s];
        if (is_group_row(v)) {
            // one record per row, for the group launch
            if (L.items_g.size() + size_t(v.R) >= static_cast<size_t>(INT32_MAX))
                return BSM_ERR_UNSUPPORTED;
            long_rows += v.R;
            for (int32_t r = 0; r < v.R; ++r)
                L.items_g.push_back({v.off + int64_t(r) * v.C, v.C, 1, r, v.R});
            ++s;
            continue;
        }
        size_t e = s + 1;
        if (spanning && v.R > 0) {
            while (e < slices.size() && slices[e].R == v.R && slices[e].C == v.C &&
                   slices[e].off == slices[e - 1].off + int64_t(v.R) * v.C) {
                slice_first[e] = static_cast<int32_t>(items.size());
                slice_first1[e] = static_cast<int32_t>(items1.size());
                L.slice_first_g[e] = static_cast<int32_t>(L.items_g.size());
                ++e;
            }
        }
        if (v.R > 0 && int64_t(v.C) * es > stage / in_arrays) {
            const int64_t seg_rows = int64_t(v.R) * static_cast<int64_t>(e - s);
            long_rows += seg_rows;
            const int64_t nch = (v.C + chunk_elems - 1) / chunk_elems;
            const int64_t per_row = std::min<int64_t>(nch, want_segs);
            const int64_t seg_elems = (nch + per_row - 1) / per_row * chunk_elems;
            const int64_t n_seg = (v.C + seg_elems - 1) / seg_elems;
            if (segs.size() < items.size())
                segs.resize(items.size(), LongSeg{0, 0, 0, 0});
            for (int64_t g = 0; g < seg_rows; ++g) {
                if (items.size() + n_seg >= static_cast<size_t>(INT32_MAX) || n_parts + n_seg >= INT32_MAX)
                    return BSM_ERR_UNSUPPORTED;
                for (int64_t k = 0; k < n_seg; ++k) {
                    const int64_t c0 = k * seg_elems;
                    const Item it{v.off + g * v.C + c0, static_cast<int32_t>(std::min<int64_t>(seg_elems, v.C - c0)),
                                  1, static_cast<int32_t>(g % v.R), v.R};
                    if (n_seg == 1) {       // the whole row, both passes in one launch
                        items.push_back(it);
                        segs.push_back(LongSeg{0, 0, 0, 1});
                        continue;
                    }
                    const LongSeg sg{static_cast<int32_t>(c0), static_cast<int32_t>(n_parts + k),
                                     static_cast<int32_t>(n_parts), static_cast<int32_t>(n_seg)};
                    items.push_back(it);
                    segs.push_back(sg);
                    items1.push_back(it);
                    segs1.push_back(sg);
                }
                if (n_seg > 1)
                    n_parts += n_seg;
            }
        } else if (v.R > 0) {
            const int64_t seg_rows = int64_t(v.R) * static_cast<int64_t>(e - s);
            const int64_t row_bytes = int64_t(v.C) * es;
            int64_t rpi = std::max<int64_t>(1, stage / in_arrays / row_bytes);
            if (d->rows_per_item > 0)
                rpi = std::min<int64_t>(rpi, d->rows_per_item);
            if (d->policy == BSM_POLICY_WHOLE_GPU)
                rpi = std::min<int64_t>(rpi, (v.R + n_sm - 1) / n_sm);
            if (spanning)
                rpi = std::min<int64_t>(rpi, spread_rows);
            rpi = std::max<int64_t>(1, std::min<int64_t>(rpi, seg_rows));
            for (int64_t g0 = 0; g0 < seg_rows; g0 += rpi) {
                if (items.size() >= static_cast<size_t>(INT32_MAX))
                    return BSM_ERR_UNSUPPORTED;
                const int64_t nr = std::min<int64_t>(rpi, seg_rows - g0);
                items.push_back({v.off + g0 * v.C, v.C, static_cast<int32_t>(nr),
                                 static_cast<int32_t>(g0 % v.R), v.R});
            }
        }
        s = e;
    }
    slice_first[slices.size()] = static_cast<int32_t>(items.size());
    slice_first1[slices.size()] = static_cast<int32_t>(items1.size());
    L.slice_first_g[slices.size()] = static_cast<int32_t>(L.items_g.size());
    if (!segs.empty())
        segs.resize(items.size(), LongSeg{0, 0, 0, 0});
    if (spanning && !items1.empty()) {
        // phase 1 takes the segments in reverse: it starts with those phase 0
        // read last, which are most likely still in L2
        std::reverse(items1.begin(), items1.end());
        std::reverse(segs1.begin(), segs1.end());
    }
    return BSM_OK;
}

// WHOLE_GPU runs one kernel per slice, one after another (Sec. 3): a
// launch-bound loop.  Plans of up to this many launches capture it once, at
// creation, as a CUDA graph, so an execute is one graph launch (the kernels
// still run in slice order, each on the whole device); larger plans launch
// kernel by kernel.
constexpr size_t kMaxGraphLaunches = 4096;

cudaGraphExec_t capture_whole_gpu(const bsm_plan *p)
{
    cudaStream_t st = nullptr;
    if (cudaStreamCreateWithFlags(&st, cudaStreamNonBlocking) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    cudaGraph_t g = nullptr;
    cudaGraphExec_t e = nullptr;
    bool ok = cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal) == cudaSuccess;
    if (ok) {
        KernelArgs a = p->args, a1 = p->args1, ag = p->argsg;
        for (const auto &l : p->whole_gpu) {
            KernelArgs &al = l.phase == 2 ? ag : (l.phase ? a1 : a);
            al.item_begin = l.begin;
            al.item_end = l.end;
            if (launch_softmax(al, p->dtype, l.phase == 2 ? OP_FORWARD_GROUP : p->kernel_op, l.grid, st, false)) {
                ok = false;
                break;
            }
        }
        const cudaError_t ec = cudaStreamEndCapture(st, &g);   // always ends the capture
        ok = ok && ec == cudaSuccess && g != nullptr;
    }
    if (ok && cudaGraphInstantiate(&e, g, 0) != cudaSuccess)
        e = nullptr;
    if (g)
        cudaGraphDestroy(g);
    cudaStreamDestroy(st);
    cudaGetLastError();   // a failed capture leaves plain launches, not an error
    return e;
}

void free_plan(bsm_plan *p)
{
    if (!p)
        return;
    if (p->whole_graph) {
        // the graph may still be running: let the plan's device finish first
        int prev = -1;
        cudaGetDevice(&prev);
        cudaSetDevice(p->device);
        cudaDeviceSynchronize();
        cudaGraphExecDestroy(p->whole_graph);
        if (prev >= 0)
            cudaSetDevice(prev);
    }
    cudaFree(p->blob);
    delete p;
}

int plan_create_impl(bsm_plan **out, const bsm_plan_desc *d)
{
    TraceRange trace("bsm_plan_create");
    const auto t0 = std::chrono::steady_clock::now();
    if (!out || !d)
        return BSM_ERR_INVALID_ARG;
    *out = nullptr;
    DeviceCtx *c = nullptr;
    int rc = device_ctx(d->device, &c);
    if (rc)
        return rc;
    int device = d->device;
    if (device < 0)
        cudaGetDevice(&device);
    std::vector<SliceView> slices;
    int64_t total = 0, max_row = 0;
    if ((rc = validate(d, slices, total, max_row)))
        return rc;
    const int es = esize(d->dtype);
    PatchLayout lay;
    if ((rc = cut_patches(d, slices, max_row, c->n_sm, c->smem_optin, lay)))
        return rc;
    const int64_t stage = lay.stage;
    const int n_stages = lay.n_stages;
    std::vector<Item> &items = lay.items;
    std::vector<LongSeg> &segs = lay.segs;
    const std::vector<Item> &items1 = lay.items1;
    const std::vector<LongSeg> &segs1 = lay.segs1;
    const std::vector<int32_t> &slice_first = lay.slice_first;
    const std::vector<int32_t> &slice_first1 = lay.slice_first1;
    const int64_t n_parts = lay.n_parts;
    const int64_t long_rows = lay.long_rows;
    // the schedule covers every patch: the regular ones, then the rows split
    // over groups of CTAs (bsm_plan_layout_host's phase-0 order)
    std::vector<Item> &items_g = lay.items_g;
    const int64_t n_reg = static_cast<int64_t>(items.size());
    const int64_t n_grp = static_cast<int64_t>(items_g.size());
    const int64_t n_items = n_reg + n_grp;
    std::vector<Item> all(items);
    all.insert(all.end(), items_g.begin(), items_g.end());

    bsm_plan *p = new bsm_plan();
    p->device = device;
    p->policy = d->policy;
    p->dtype = d->dtype;
    p->op = d->op;
    p->x = d->x;
    p->y = d->y;
    p->flags = d->flags;
    bsm_plan_stats &st = p->stats;
    std::memset(&st, 0, sizeof st);
    st.policy = d->policy;
    st.n_die = 1;
    st.n_items = n_items;
    st.stage_bytes = static_cast<int32_t>(stage);
    st.n_stages = n_stages;
    st.long_items = long_rows;
    st.group_rows = n_grp;
    st.group_k = lay.group_k;
    st.n_groups = n_grp ? lay.n_groups : 0;
    const bool reg_long = long_rows > n_grp;   // long rows outside the groups
    p->kernel_op = d->op == BSM_OP_BACKWARD ? (reg_long ? OP_BACKWARD_LONG : OP_BACKWARD)
                                            : (reg_long ? OP_FORWARD_LONG : OP_FORWARD);

    // ---- the schedule
    std::vector<int32_t> queue;      // schedule order of the patches (queue policies)
    int32_t qbeg[BSM_MAX_DIES] = {0}, qlen[BSM_MAX_DIES] = {0};
    int n_queues = 1;
    int8_t sm_die_tab[BSM_MAX_SM];
    std::memset(sm_die_tab, 0, sizeof sm_die_tab);
    bool use_sm_die = false;
    if (d->policy == BSM_POLICY_DYNAMIC) {
        queue.resize(static_cast<size_t>(n_items));
        std::iota(queue.begin(), queue.end(), 0);
        qlen[0] = static_cast<int32_t>(n_items);
        st.queue_items[0] = n_items;
        st.queue_bytes[0] = total * es * 2;
        st.L[0] = st.N[0] = n_items;
    } else if (d->policy == BSM_POLICY_CBMF || d->policy == BSM_POLICY_CBMF_LB ||
               d->policy == BSM_POLICY_MINIMAX) {
        bsm_topology topo;
        if ((rc = topology_get(device, 0, &topo))) {
            delete p;
            return rc;
        }
        const bool lb = d->policy == BSM_POLICY_CBMF_LB;
        const bool minimax = d->policy == BSM_POLICY_MINIMAX;
        if (!topo.separable || n_items == 0) {
            // one die: CBMF degenerates to a single queue
            queue.resize(static_cast<size_t>(n_items));
            std::iota(queue.begin(), queue.end(), 0);
            qlen[0] = static_cast<int32_t>(n_items);
            st.queue_items[0] = n_items;
            st.L[0] = st.N[0] = n_items;
        } else {
            const int nb = 2;
            const int64_t xbytes = total * es;
            int64_t chunk = std::max<int64_t>(128, topo.granularity);
            chunk = (chunk + 127) & ~int64_t(127);
            while ((xbytes + chunk - 1) / chunk > kMaxMapChunks)
                chunk *= 2;
            st.map_chunk_bytes = chunk;
            const int64_t nch = (xbytes + chunk - 1) / chunk;
            std::vector<int8_t> xmap(static_cast<size_t>(nch)), ymap;
            if ((rc = addr_die_map_host(device, d->x, xbytes, chunk, xmap.data()))) {
                delete p;
                return rc;
            }
            const bool count_y = d->count_output_bytes != 0;
            if (count_y) {
                if (d->y == d->x) {
                    ymap = xmap;
                } else {
                    ymap.resize(static_cast<size_t>(nch));
                    if ((rc = addr_die_map_host(device, d->y, xbytes, chunk, ymap.data()))) {
                        delete p;
                        return rc;
                    }
                }
            }
            std::vector<int64_t> pb(static_cast<size_t>(n_items)), pe(static_cast<size_t>(n_items)),
                cost(static_cast<size_t>(n_items));
            for (int64_t i = 0; i < n_items; ++i) {
                pb[i] = all[i].off * es;
                pe[i] = (all[i].off + int64_t(all[i].nrows) * all[i].C) * es;
                cost[i] = 2 * (pe[i] - pb[i]);
            }
            int32_t units[BSM_MAX_DIES] = {std::max(1, topo.sm_per_die[0]), std::max(1, topo.sm_per_die[1])};
            bsm_schedule_desc sd{};
            sd.n_banks = nb;
            sd.n_patches = n_items;
            sd.patch_begin = pb.data();
            sd.patch_end = pe.data();
            sd.n_maps = count_y ? 2 : 1;
            sd.chunk[0] = sd.chunk[1] = chunk;
            sd.n_chunks[0] = sd.n_chunks[1] = nch;
            sd.bank_of_chunk[0] = xmap.data();
            sd.bank_of_chunk[1] = count_y ? ymap.data() : nullptr;
            sd.tie_seed = d->tie_seed;
            sd.balance = lb ? 1 : 0;
            sd.method = minimax ? 1 : 0;
            sd.units = units;
            sd.l_near = d->lb_weighted ? std::max<int64_t>(1, llround(topo.l_near)) : 1;
            sd.l_far = d->lb_weighted ? std::max<int64_t>(1, llround(topo.l_far)) : 1;
            sd.cost = cost.data();
            std::vector<int64_t> bob(static_cast<size_t>(n_items) * nb);
            std::vector<uint8_t> ov(static_cast<size_t>(n_items));
            std::vector<int32_t> bank(static_cast<size_t>(n_items)), qi(static_cast<size_t>(n_items)),
                moved(static_cast<size_t>(n_items));
            int64_t N[BSM_MAX_DIES] = {0}, L[BSM_MAX_DIES] = {0}, ql[BSM_MAX_DIES] = {0};
            int64_t wb[BSM_MAX_DIES] = {0}, wa[BSM_MAX_DIES] = {0};
            bsm_schedule_out so{};
            so.bytes_on_bank = bob.data();
            so.overlap = ov.data();
            so.N = N;
            so.bank = bank.data();
            so.L = L;
            so.queue_items = qi.data();
            so.queue_len = ql;
            so.moved = moved.data();
            so.work_before = wb;
            so.work_after = wa;
            if ((rc = schedule_host(&sd, &so))) {
                delete p;
                return rc;
            }
            queue = qi;
            p->xmap = xmap;
            p->ymap = count_y && d->y != d->x ? ymap : std::vector<int8_t>();
            p->map_chunk = chunk;
            p->moved.assign(moved.begin(), moved.begin() + so.n_moved);
            for (int b = 0; b < nb; ++b)
                p->units[b] = units[b];
            p->w_near = sd.l_near;
            p->w_far = sd.l_far;
            p->count_y = count_y ? 1 : 0;
            p->tie_seed = d->tie_seed;
            n_queues = nb;
            int32_t pos = 0;
            for (int b = 0; b < nb; ++b) {
                qbeg[b] = pos;
                qlen[b] = static_cast<int32_t>(ql[b]);
                pos += qlen[b];
                st.N[b] = N[b];
                st.L[b] = L[b];
                st.queue_items[b] = ql[b];
                int64_t bytes = 0;
                for (int32_t k = qbeg[b]; k < qbeg[b] + qlen[b]; ++k)
                    bytes += cost[queue[k]];
                st.queue_bytes[b] = bytes;
                if (lb) {
                    st.est_finish_before[b] = double(wb[b]) / units[b];
                    st.est_finish_after[b] = double(wa[b]) / units[b];
                } else if (minimax) {
                    st.est_finish_after[b] = double(wa[b]) / units[b];
                }
            }
            for (int64_t i = 0; i < n_items; ++i) {
                st.overlap_items += ov[i];
                const int64_t *row = &bob[static_cast<size_t>(i) * nb];
                if (row[0] == row[1])
                    ++st.tie_items;
            }
            st.moved_items = so.n_moved;
            st.n_die = nb;
            std::memcpy(sm_die_tab, topo.sm_die, sizeof sm_die_tab);
            for (int sm = 0; sm < BSM_MAX_SM; ++sm)
                if (sm_die_tab[sm] < 0)
                    sm_die_tab[sm] = 0;
            use_sm_die = true;
            p->args.steal = (lb || minimax) ? 1 : 0;
        }
    }

    p->queue = queue;
    p->q_count = queue.empty() ? 0 : n_queues;
    for (int b = 0; b < BSM_MAX_DIES; ++b) {
        p->q_begin[b] = qbeg[b];
        p->q_len[b] = qlen[b];
    }
    // ---- queue policies store the patches in queue order (die 0's queue,
    // then die 1's, ...), so a claimed queue slot is the patch record itself;
    // the regular patches and the group rows go to tables of their own, each
    // in that order
    int32_t qbeg_g[BSM_MAX_DIES] = {0}, qlen_g[BSM_MAX_DIES] = {0};
    if (!queue.empty()) {
        std::vector<Item> ordered, ordered_g;
        std::vector<LongSeg> osegs;
        ordered.reserve(items.size());
        ordered_g.reserve(items_g.size());
        for (int b = 0; b < n_queues; ++b) {
            const int32_t r0 = static_cast<int32_t>(ordered.size()), g0 = static_cast<int32_t>(ordered_g.size());
            for (int32_t k = qbeg[b]; k < qbeg[b] + qlen[b]; ++k) {
                const int64_t i = queue[static_cast<size_t>(k)];
                if (i < n_reg) {
                    ordered.push_back(items[static_cast<size_t>(i)]);
                    if (!segs.empty())
                        osegs.push_back(segs[static_cast<size_t>(i)]);
                } else {
                    ordered_g.push_back(items_g[static_cast<size_t>(i - n_reg)]);
                }
            }
            qbeg[b] = r0;
            qlen[b] = static_cast<int32_t>(ordered.size()) - r0;
            qbeg_g[b] = g0;
            qlen_g[b] = static_cast<int32_t>(ordered_g.size()) - g0;
        }
        items.swap(ordered);
        items_g.swap(ordered_g);
        if (!segs.empty())
            segs.swap(osegs);
    }

    // ---- upload the tables in one allocation
    const size_t items_b = sizeof(Item) * items.size();          // the regular patches only
    const size_t slices_b = sizeof(int32_t) * slice_first.size();
    const int64_t n1 = static_cast<int64_t>(items1.size());
    const size_t segs_b = sizeof(LongSeg) * segs.size(), items1_b = sizeof(Item) * items1.size(),
                 segs1_b = sizeof(LongSeg) * segs1.size(), parts_b = 2 * sizeof(float) * size_t(n_parts);
    auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
    const int64_t gk = lay.group_k, gn = n_grp ? lay.n_groups : 0;
    const size_t itemsg_b = sizeof(Item) * items_g.size(), ring_b = sizeof(uint64_t) * kGroupRing * size_t(gn),
                 xch_b = 2 * sizeof(uint64_t) * kGroupSlots * size_t(gn * gk);
    const size_t o_items = 0, o_slices = up(items_b), o_smdie = o_slices + up(slices_b),
                 o_heads = o_smdie + 256, o_segs = o_heads + 256, o_items1 = o_segs + up(segs_b),
                 o_segs1 = o_items1 + up(items1_b), o_slices1 = o_segs1 + up(segs1_b),
                 o_heads1 = o_slices1 + (n1 ? up(slices_b) : 0), o_parts = o_heads1 + 256,
                 o_itemsg = o_parts + up(parts_b), o_slicesg = o_itemsg + up(itemsg_b),
                 o_headsg = o_slicesg + (n_grp ? up(slices_b) : 0), o_ring = o_headsg + 256,
                 o_xch = o_ring + up(ring_b), blob_b = o_xch + up(xch_b);
    std::vector<unsigned char> host(blob_b, 0);
    if (n_grp) {
        std::memcpy(&host[o_itemsg], items_g.data(), itemsg_b);
        std::memcpy(&host[o_slicesg], lay.slice_first_g.data(), slices_b);
    }
    if (items_b)
        std::memcpy(&host[o_items], items.data(), items_b);
    std::memcpy(&host[o_slices], slice_first.data(), slices_b);
    std::memcpy(&host[o_smdie], sm_die_tab, BSM_MAX_SM);
    if (segs_b)
        std::memcpy(&host[o_segs], segs.data(), segs_b);
    if (n1) {
        std::memcpy(&host[o_items1], items1.data(), items1_b);
        std::memcpy(&host[o_segs1], segs1.data(), segs1_b);
        std::memcpy(&host[o_slices1], slice_first1.data(), slices_b);
    }
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(device);
    if (cudaMalloc(&p->blob, blob_b) != cudaSuccess) {
        if (prev >= 0)
            cudaSetDevice(prev);
        delete p;
        return BSM_ERR_NOMEM;
    }
    if (cudaError_t e = cudaMemcpy(p->blob, host.data(), blob_b, cudaMemcpyHostToDevice)) {
        cudaFree(p->blob);
        if (prev >= 0)
            cudaSetDevice(prev);
        delete p;
        return cuda_error(e, "cudaMemcpy(plan tables)");
    }
    if (prev >= 0)
        cudaSetDevice(prev);
    unsigned char *b = static_cast<unsigned char *>(p->blob);

    KernelArgs &a = p->args;
    a.n_items = static_cast<int32_t>(n_reg);
    a.x = d->x;
    a.x2 = d->op == BSM_OP_BACKWARD ? d->x2 : nullptr;
    a.y = d->y;
    a.total_elems = total;
    a.items = reinterpret_cast<const Item *>(b + o_items);
    a.slice_first_item = reinterpret_cast<const int32_t *>(b + o_slices);
    a.n_slices = static_cast<int32_t>(std::min<size_t>(slices.size(), INT32_MAX));
    a.n_queues = n_queues;
    for (int q = 0; q < BSM_MAX_DIES; ++q) {
        a.queue_begin[q] = qbeg[q];
        a.queue_len[q] = qlen[q];
    }
    a.heads = reinterpret_cast<uint32_t *>(b + o_heads);
    a.sm_die = use_sm_die ? reinterpret_cast<const int8_t *>(b + o_smdie) : nullptr;
    a.stage_bytes = static_cast<int32_t>(stage);
    a.n_stages = n_stages;
    a.flags = d->flags;
    a.status = c->status;
    a.segs = segs.empty() ? nullptr : reinterpret_cast<const LongSeg *>(b + o_segs);
    a.partials = n_parts ? reinterpret_cast<float *>(b + o_parts) : nullptr;
    a.phase = 0;
    // phase 1 (rows longer than a stage): their segments again, one queue
    // (or the same static / round-robin split as phase 0)
    p->n_phase1 = n1;
    if (n1) {
        KernelArgs &a1 = p->args1;
        a1 = a;
        a1.items = reinterpret_cast<const Item *>(b + o_items1);
        a1.segs = reinterpret_cast<const LongSeg *>(b + o_segs1);
        a1.n_items = static_cast<int32_t>(n1);
        a1.slice_first_item = reinterpret_cast<const int32_t *>(b + o_slices1);
        a1.n_queues = 1;
        for (int q = 0; q < BSM_MAX_DIES; ++q)
            a1.queue_begin[q] = a1.queue_len[q] = 0;
        a1.queue_len[0] = static_cast<int32_t>(n1);
        a1.steal = 0;
        a1.sm_die = nullptr;
        a1.heads = reinterpret_cast<uint32_t *>(b + o_heads1);
        a1.phase = 1;
    }
    // rows over groups of CTAs: their table, queues and exchange buffers
    p->n_group = n_grp;
    if (n_grp) {
        KernelArgs &ag = p->argsg;
        ag = a;
        ag.items = reinterpret_cast<const Item *>(b + o_itemsg);
        ag.n_items = static_cast<int32_t>(n_grp);
        ag.slice_first_item = reinterpret_cast<const int32_t *>(b + o_slicesg);
        for (int q = 0; q < BSM_MAX_DIES; ++q) {
            ag.queue_begin[q] = queue.empty() ? 0 : qbeg_g[q];
            ag.queue_len[q] = queue.empty() ? 0 : qlen_g[q];
        }
        ag.heads = reinterpret_cast<uint32_t *>(b + o_headsg);
        // a group pulls from the die queue of its rank-0 CTA's SM, and from
        // the other die's once that is empty -- also under CBMF: the groups
        // (a group may span both dies) need not cover both dies, and every
        // queue must be drained
        if (ag.n_queues > 1)
            ag.steal = 1;
        ag.stage_bytes = static_cast<int32_t>(lay.stage_g);
        ag.n_stages = lay.n_stages_g;
        ag.segs = nullptr;
        ag.partials = nullptr;
        ag.phase = 0;
        ag.group_k = lay.group_k;
        ag.n_groups = lay.n_groups;
        ag.ring = reinterpret_cast<unsigned long long *>(b + o_ring);
        ag.xch = reinterpret_cast<unsigned long long *>(b + o_xch);
        p->grid_g = lay.group_k * lay.n_groups;
    }

    const int32_t other_launches = (n_reg > 0 ? (n1 ? 2 : 1) : 0) + (n_grp > 0 ? 1 : 0);
    switch (d->policy) {
    case BSM_POLICY_WHOLE_GPU:
        a.mode = PULL_STATIC;
        for (size_t k = 0; k < slices.size(); ++k) {
            const int32_t n = slice_first[k + 1] - slice_first[k];
            if (n > 0)
                p->whole_gpu.push_back({slice_first[k], slice_first[k + 1], std::min(n, c->n_sm), 0});
            const int32_t n1s = slice_first1[k + 1] - slice_first1[k];
            if (n1s > 0)
                p->whole_gpu.push_back({slice_first1[k], slice_first1[k + 1], std::min(n1s, c->n_sm), 1});
            if (n_grp) {
                const int32_t ng = lay.slice_first_g[k + 1] - lay.slice_first_g[k];
                if (ng > 0)
                    p->whole_gpu.push_back({lay.slice_first_g[k], lay.slice_first_g[k + 1], p->grid_g, 2});
            }
        }
        p->grid = c->n_sm;
        st.launches = static_cast<int32_t>(p->whole_gpu.size());
        break;
    case BSM_POLICY_RR:
        a.mode = PULL_RR_SLICE;
        p->grid = static_cast<int>(std::min<int64_t>(c->n_sm, std::max<int64_t>(1, int64_t(slices.size()))));
        st.launches = other_launches;
        break;
    default:
        a.mode = PULL_QUEUE;
        p->grid = c->n_sm;
        st.launches = other_launches;
        break;
    }
    p->args1.mode = a.mode;
    p->argsg.mode = a.mode;
    // one queue no longer than the grid (a small batch: a patch per SM at
    // most): CTA u takes queue slot u and nothing else, with no claim before
    // its copy and no queue head to rewind after it -- the static deal over
    // the queue's slots
    if (a.mode == PULL_QUEUE && a.n_queues == 1 && a.queue_len[0] <= p->grid) {
        a.mode = PULL_STATIC;
        a.item_begin = a.queue_begin[0];
        a.item_end = a.queue_begin[0] + a.queue_len[0];
    }
    // (rows over groups of CTAs use cooperative launches, which stay out of
    // the graph: such plans launch kernel by kernel)
    if (d->policy == BSM_POLICY_WHOLE_GPU && !p->whole_gpu.empty() && p->whole_gpu.size() <= kMaxGraphLaunches &&
        n_grp == 0) {
        int prev_dev = -1;
        cudaGetDevice(&prev_dev);
        cudaSetDevice(device);
        p->whole_graph = capture_whole_gpu(p);
        if (prev_dev >= 0)
            cudaSetDevice(prev_dev);
    }
    st.grid = p->grid;
    st.steal = a.steal;
    st.plan_ms = std::chrono::duration<double, std::milli>(std::chrono::steady_clock::now() - t0).count();
    *out = p;
    return BSM_OK;
}

int plan_layout_host_impl(const bsm_plan_desc *d, int32_t n_sm, int64_t smem_optin, bsm_patch *phase0,
                          int64_t cap0, bsm_patch *phase1, int64_t cap1, bsm_layout *out)
{
    if (!d || !out || n_sm < 1 || n_sm > BSM_MAX_SM || smem_optin <= kSmemHeader ||
        smem_optin > (int64_t(1) << 20) || cap0 < 0 || cap1 < 0 || (cap0 > 0 && !phase0) ||
        (cap1 > 0 && !phase1))
        return BSM_ERR_INVALID_ARG;
    std::memset(out, 0, sizeof *out);
    std::vector<SliceView> slices;
    int64_t total = 0, max_row = 0;
    int rc = validate(d, slices, total, max_row);
    if (rc)
        return rc;
    PatchLayout lay;
    if ((rc = cut_patches(d, slices, max_row, n_sm, smem_optin, lay)))
        return rc;
    out->stage_bytes = lay.stage;
    out->n_stages = lay.n_stages;
    out->group_k = lay.items_g.empty() ? 0 : lay.group_k;
    out->n_patches = static_cast<int64_t>(lay.items.size() + lay.items_g.size());
    out->n_patches_phase1 = static_cast<int64_t>(lay.items1.size());
    out->long_rows = lay.long_rows;
    auto put = [](const Item &it, const LongSeg *sg, bsm_patch &o) {
        o.elem_offset = it.off;
        o.cols = it.C;
        o.nrows = it.nrows;
        o.row0 = it.row0;
        o.slice_rows = it.R;
        o.col0 = sg ? sg->col0 : 0;
        o.part_count = sg ? sg->part_count : 0;
    };
    for (size_t i = 0; i < lay.items.size() && static_cast<int64_t>(i) < cap0; ++i)
        put(lay.items[i], lay.segs.empty() ? nullptr : &lay.segs[i], phase0[i]);
    // rows over groups of CTAs come last, marked part_count = -K
    for (size_t j = 0; j < lay.items_g.size() && static_cast<int64_t>(lay.items.size() + j) < cap0; ++j) {
        bsm_patch &o = phase0[lay.items.size() + j];
        put(lay.items_g[j], nullptr, o);
        o.part_count = -lay.group_k;
    }
    for (size_t i = 0; i < lay.items1.size() && static_cast<int64_t>(i) < cap1; ++i)
        put(lay.items1[i], &lay.segs1[i], phase1[i]);
    return BSM_OK;
}

int plan_execute_impl(const bsm_plan *p, bsm_stream_t stream)
{
    TraceRange trace("bsm_plan_execute");
    if (!p)
        return BSM_ERR_INVALID_ARG;
    if (p->args.n_items == 0 && p->n_group == 0)
        return BSM_OK;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != p->device && cudaSetDevice(p->device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    int err = 0;
    const bool checked = g_checked.load(std::memory_order_relaxed) != 0;
    if (p->policy == BSM_POLICY_WHOLE_GPU && p->whole_graph && !checked && p->args.debug == 0 &&
        p->args.wait_limit_ns == 0) {
        err = static_cast<int>(cudaGraphLaunch(p->whole_graph, static_cast<cudaStream_t>(stream)));
    } else if (p->policy == BSM_POLICY_WHOLE_GPU) {
        KernelArgs a = p->args, a1 = p->args1, ag = p->argsg;
        for (const auto &l : p->whole_gpu) {
            KernelArgs &al = l.phase == 2 ? ag : (l.phase ? a1 : a);
            al.item_begin = l.begin;
            al.item_end = l.end;
            if ((err = launch_softmax(al, p->dtype, l.phase == 2 ? OP_FORWARD_GROUP : p->kernel_op, l.grid, stream,
                                      checked)))
                break;
        }
    } else {
        if (p->args.n_items > 0)
            err = launch_softmax(p->args, p->dtype, p->kernel_op, p->grid, stream, checked);
        if (!err && p->n_phase1)
            err = launch_softmax(p->args1, p->dtype, p->kernel_op, p->grid, stream, checked);
        if (!err && p->n_group)
            err = launch_softmax(p->argsg, p->dtype, OP_FORWARD_GROUP, p->grid_g, stream, checked);
    }
    if (prev >= 0 && prev != p->device)
        cudaSetDevice(prev);
    return err ? cuda_error(static_cast<cudaError_t>(err), "kernel launch") : BSM_OK;
}

// ---- plan cache of the one-call entry points

struct CacheKey {
    int device;
    const void *x;
    void *y;
    int dtype, policy;
    uint32_t flags;
    int op;
    const void *x2;
};

std::mutex g_cache_mu;
std::list<bsm_plan *> g_cache;   // most recent first
constexpr size_t kCacheMax = 32;

bool same_key(const bsm_plan *p, const CacheKey &k)
{
    return p->device == k.device && p->x == k.x && p->y == k.y && p->dtype == k.dtype &&
           p->policy == k.policy && p->flags == k.flags && p->op == k.op && p->args.x2 == k.x2;
}

int cached_run(const CacheKey &k, int64_t B, int64_t R, int64_t C, int64_t n, const int64_t *off,
               const int32_t *rows, const int32_t *cols, bsm_stream_t stream)
{
    std::lock_guard<std::mutex> lk(g_cache_mu);
    for (auto it = g_cache.begin(); it != g_cache.end(); ++it) {
        bsm_plan *p = *it;
        if (!same_key(p, k))
            continue;
        bool hit;
        if (B >= 0) {
            hit = p->key_B == B && p->key_R == R && p->key_C == C;
        } else {
            hit = p->key_B < 0 && static_cast<int64_t>(p->key_rows.size()) == n &&
                  std::equal(rows, rows + n, p->key_rows.begin()) &&
                  std::equal(cols, cols + n, p->key_cols.begin()) &&
                  std::equal(off, off + n, p->key_offsets.begin());
        }
        if (hit) {
            g_cache.splice(g_cache.begin(), g_cache, it);
            return plan_execute_impl(p, stream);
        }
    }
    bsm_plan_desc d;
    bsm_plan_desc_init(&d);
    d.x = k.x;
    d.y = k.y;
    d.dtype = k.dtype;
    d.policy = k.policy;
    d.flags = k.flags;
    d.device = k.device;
    d.op = k.op;
    d.x2 = k.x2;
    std::vector<int32_t> r, c;
    if (B >= 0) {
        if (B > INT32_MAX || R > INT32_MAX || C > INT32_MAX)
            return BSM_ERR_UNSUPPORTED;
        r.assign(static_cast<size_t>(B), static_cast<int32_t>(R));
        c.assign(static_cast<size_t>(B), static_cast<int32_t>(C));
        d.num_slices = B;
        d.rows = r.data();
        d.cols = c.data();
    } else {
        d.num_slices = n;
        d.offsets = off;
        d.rows = rows;
        d.cols = cols;
    }
    bsm_plan *p = nullptr;
    int rc = plan_create_impl(&p, &d);
    if (rc)
        return rc;
    if (B >= 0) {
        p->key_B = B;
        p->key_R = R;
        p->key_C = C;
    } else {
        p->key_offsets.assign(off, off + n);
        p->key_rows.assign(rows, rows + n);
        p->key_cols.assign(cols, cols + n);
    }
    g_cache.push_front(p);
    while (g_cache.size() > kCacheMax) {
        bsm_plan *old = g_cache.back();
        g_cache.pop_back();
        free_plan(old);
    }
    return plan_execute_impl(p, stream);
}

}  // namespace
}  // namespace bsm

using namespace bsm;

#define BSM_GUARD(expr)                                  \
    try {                                                \
        return (expr);                                   \
    } catch (const std::bad_alloc &) {                   \
        return BSM_ERR_NOMEM;                            \
    } catch (...) {                                      \
        return BSM_ERR_INVALID_ARG;                      \
    }

extern "C" {

int bsm_plan_desc_init(bsm_plan_desc *d)
{
    if (!d)
        return BSM_ERR_INVALID_ARG;
    std::memset(d, 0, sizeof *d);
    d->tie_seed = kDefaultTieSeed;
    d->lb_weighted = 1;
    d->count_output_bytes = 1;
    d->device = -1;
    return BSM_OK;
}

int bsm_plan_create(bsm_plan **plan, const bsm_plan_desc *d) { BSM_GUARD(plan_create_impl(plan, d)) }

int bsm_plan_execute(const bsm_plan *plan, bsm_stream_t stream) { BSM_GUARD(plan_execute_impl(plan, stream)) }

int bsm_plan_get_stats(const bsm_plan *plan, bsm_plan_stats *out)
{
    if (!plan || !out)
        return BSM_ERR_INVALID_ARG;
    *out = plan->stats;
    return BSM_OK;
}

int bsm_plan_get_schedule(const bsm_plan *plan, bsm_plan_schedule *out)
{
    if (!plan || !out)
        return BSM_ERR_INVALID_ARG;
    const bsm_plan &p = *plan;
    const bool queued = p.q_count > 0;
    out->n_queues = p.q_count;
    out->count_output_bytes = p.count_y;
    for (int b = 0; b < BSM_MAX_DIES; ++b) {
        out->queue_begin[b] = queued ? p.q_begin[b] : 0;
        out->queue_len[b] = queued ? p.q_len[b] : 0;
        out->units[b] = p.units[b];
    }
    out->l_near = p.w_near;
    out->l_far = p.w_far;
    out->tie_seed = p.tie_seed;
    out->n_items = p.stats.n_items;
    out->map_chunk_bytes = p.map_chunk;
    out->n_map_chunks = static_cast<int64_t>(p.xmap.size());
    out->n_moved = static_cast<int64_t>(p.moved.size());
    if (out->queue && queued)
        std::memcpy(out->queue, p.queue.data(), sizeof(int32_t) * p.queue.size());
    if (out->x_map && !p.xmap.empty())
        std::memcpy(out->x_map, p.xmap.data(), p.xmap.size());
    if (out->y_map && !p.ymap.empty())
        std::memcpy(out->y_map, p.ymap.data(), p.ymap.size());
    if (out->moved && !p.moved.empty())
        std::memcpy(out->moved, p.moved.data(), sizeof(int32_t) * p.moved.size());
    return BSM_OK;
}

int bsm_plan_device_table(const bsm_plan *plan, int phase, bsm_patch *out, int64_t cap, int64_t *n_out)
{
    if (!plan || !n_out || phase < 0 || phase > 2 || cap < 0 || (cap > 0 && !out))
        return BSM_ERR_INVALID_ARG;
    const KernelArgs &a = phase == 2 ? plan->argsg : (phase ? plan->args1 : plan->args);
    const int64_t n = (phase == 1 && !plan->n_phase1) || (phase == 2 && !plan->n_group) ? 0 : a.n_items;
    *n_out = n;
    const int64_t m = std::min(n, cap);
    if (m <= 0)
        return BSM_OK;
    std::vector<Item> items(static_cast<size_t>(m));
    std::vector<LongSeg> segs;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(plan->device);
    cudaError_t e = cudaMemcpy(items.data(), a.items, sizeof(Item) * items.size(), cudaMemcpyDeviceToHost);
    if (e == cudaSuccess && a.segs) {
        segs.resize(static_cast<size_t>(m));
        e = cudaMemcpy(segs.data(), a.segs, sizeof(LongSeg) * segs.size(), cudaMemcpyDeviceToHost);
    }
    if (prev >= 0)
        cudaSetDevice(prev);
    if (e != cudaSuccess)
        return cuda_error(e, "cudaMemcpy(plan table)");
    for (int64_t i = 0; i < m; ++i) {
        out[i].elem_offset = items[i].off;
        out[i].cols = items[i].C;
        out[i].nrows = items[i].nrows;
        out[i].row0 = items[i].row0;
        out[i].slice_rows = items[i].R;
        out[i].col0 = segs.empty() ? 0 : segs[i].col0;
        out[i].part_count = phase == 2 ? -a.group_k : (segs.empty() ? 0 : segs[i].part_count);
    }
    return BSM_OK;
}

int bsm_die_check_read(int device, const void *ptr, int64_t bytes, int64_t chunk, const int8_t *die_of_chunk,
                       const int8_t *sm_group, int invert, uint32_t *xor_out, float *ms_out)
{
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    BSM_GUARD(die_check_host(device, ptr, bytes, chunk, die_of_chunk, sm_group, invert, xor_out, ms_out))
}

int bsm_addr_group_map(int device, const void *ptr, int64_t bytes, int64_t chunk, const int8_t *sm_group,
                       int8_t *group_out)
{
    if (!sm_group)
        return BSM_ERR_INVALID_ARG;
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    BSM_GUARD(addr_die_map_host(device, ptr, bytes, chunk, group_out, sm_group))
}

int bsm_plan_debug(bsm_plan *plan, int what, int64_t arg)
{
    if (!plan)
        return noalloc_debug(what, arg);
    switch (what) {
    case BSM_DEBUG_NONE:
        plan->args.debug = 0;
        plan->args.wait_limit_ns = 0;
        plan->args1.debug = 0;
        plan->args1.wait_limit_ns = 0;
        plan->argsg.debug = 0;
        plan->argsg.wait_limit_ns = 0;
        return BSM_OK;
    case BSM_DEBUG_WITHHOLD_STAGE:
        if (arg <= 0)
            return BSM_ERR_INVALID_ARG;
        plan->args.debug |= KDEBUG_WITHHOLD_STAGE0;
        plan->args.wait_limit_ns = static_cast<uint64_t>(arg);
        plan->argsg.debug |= KDEBUG_WITHHOLD_STAGE0;
        plan->argsg.wait_limit_ns = static_cast<uint64_t>(arg);
        return BSM_OK;
    case BSM_DEBUG_CORRUPT_PATCH: {
        // slots of the regular table first, then those of the group rows
        if (arg < 0 || arg >= int64_t(plan->args.n_items) + plan->n_group)
            return BSM_ERR_INVALID_ARG;
        const int64_t past_end = plan->args.total_elems;
        unsigned char *entry =
            arg < plan->args.n_items
                ? static_cast<unsigned char *>(plan->blob) + sizeof(Item) * static_cast<size_t>(arg)
                : reinterpret_cast<unsigned char *>(const_cast<Item *>(plan->argsg.items)) +
                      sizeof(Item) * static_cast<size_t>(arg - plan->args.n_items);
        int prev = -1;
        cudaGetDevice(&prev);
        cudaSetDevice(plan->device);
        cudaError_t e = cudaMemcpy(entry + offsetof(Item, off), &past_end, sizeof past_end,
                                   cudaMemcpyHostToDevice);
        if (prev >= 0)
            cudaSetDevice(prev);
        return e == cudaSuccess ? BSM_OK : cuda_error(e, "cudaMemcpy(patch entry)");
    }
    default:
        return BSM_ERR_INVALID_ARG;
    }
}

void bsm_plan_destroy(bsm_plan *plan)
{
    bsm::free_plan(plan);
}

int bsm_plan_layout_host(const bsm_plan_desc *d, int32_t n_sm, int64_t smem_optin, bsm_patch *phase0,
                         int64_t cap0, bsm_patch *phase1, int64_t cap1, bsm_layout *out)
{
    BSM_GUARD(plan_layout_host_impl(d, n_sm, smem_optin, phase0, cap0, phase1, cap1, out))
}

void bsm_cache_clear(void)
{
    std::lock_guard<std::mutex> lk(g_cache_mu);
    for (bsm_plan *p : g_cache)
        bsm::free_plan(p);
    g_cache.clear();
}

static int softmax_uniform(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype, int policy,
                           uint32_t flags, bsm_stream_t stream, int op = BSM_OP_FORWARD,
                           const void *x2 = nullptr)
{
    if (B < 0 || R < 0 || C < 1)
        return BSM_ERR_INVALID_ARG;
    if (dtype != BSM_F32 && dtype != BSM_BF16)
        return BSM_ERR_INVALID_ARG;
    if (policy < BSM_POLICY_WHOLE_GPU || policy > BSM_POLICY_MINIMAX || (flags & ~BSM_FLAG_CAUSAL))
        return BSM_ERR_INVALID_ARG;
    if (R > 0 && (B > (int64_t(1) << 62) / R || C > (int64_t(1) << 62) / std::max<int64_t>(1, B * R)))
        return BSM_ERR_INVALID_ARG;
    if (B == 0 || R == 0)
        return BSM_OK;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    CacheKey k{dev, x, y, dtype, policy, flags, op, x2};
    return cached_run(k, B, R, C, 0, nullptr, nullptr, nullptr, stream);
}

int bsm_softmax(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype, int policy,
                bsm_stream_t stream)
{
    BSM_GUARD(softmax_uniform(x, y, B, R, C, dtype, policy, 0u, stream))
}

int bsm_softmax_ex(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype, int policy,
                   uint32_t flags, bsm_stream_t stream)
{
    BSM_GUARD(softmax_uniform(x, y, B, R, C, dtype, policy, flags, stream))
}

static int softmax_ragged(const void *x, void *y, int64_t n, const int64_t *off, const int32_t *rows,
                          const int32_t *cols, int dtype, int policy, uint32_t flags, bsm_stream_t stream,
                          int op = BSM_OP_FORWARD, const void *x2 = nullptr)
{
    if (n < 0 || (n > 0 && (!off || !rows || !cols)))
        return BSM_ERR_INVALID_ARG;
    if (dtype != BSM_F32 && dtype != BSM_BF16)
        return BSM_ERR_INVALID_ARG;
    if (policy < BSM_POLICY_WHOLE_GPU || policy > BSM_POLICY_MINIMAX || (flags & ~BSM_FLAG_CAUSAL))
        return BSM_ERR_INVALID_ARG;
    if (n == 0)
        return BSM_OK;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    CacheKey k{dev, x, y, dtype, policy, flags, op, x2};
    return cached_run(k, -1, 0, 0, n, off, rows, cols, stream);
}

int bsm_softmax_ragged(const void *x, void *y, int64_t num_slices, const int64_t *offsets,
                       const int32_t *rows, const int32_t *cols, int dtype, int policy, uint32_t flags,
                       bsm_stream_t stream)
{
    BSM_GUARD(softmax_ragged(x, y, num_slices, offsets, rows, cols, dtype, policy, flags, stream))
}

int bsm_softmax_backward(const void *y, const void *dy, void *dx, int64_t B, int64_t R, int64_t C,
                         int dtype, int policy, bsm_stream_t stream)
{
    if (!dy && B > 0 && R > 0)
        return BSM_ERR_INVALID_ARG;
    BSM_GUARD(softmax_uniform(y, dx, B, R, C, dtype, policy, 0u, stream, BSM_OP_BACKWARD, dy))
}

int bsm_softmax_backward_ragged(const void *y, const void *dy, void *dx, int64_t num_slices,
                                const int64_t *offsets, const int32_t *rows, const int32_t *cols,
                                int dtype, int policy, bsm_stream_t stream)
{
    if (!dy && num_slices > 0)
        return BSM_ERR_INVALID_ARG;
    BSM_GUARD(softmax_ragged(y, dx, num_slices, offsets, rows, cols, dtype, policy, 0u, stream,
                             BSM_OP_BACKWARD, dy))
}

int bsm_topology_probe(int device, int force, bsm_topology *out)
{
    if (!out)
        return BSM_ERR_INVALID_ARG;
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    DeviceCtx *c = nullptr;
    int rc = device_ctx(device, &c);
    if (rc)
        return rc;
    BSM_GUARD(topology_get(device, force, out))
}

int bsm_addr_die_map(int device, const void *ptr, int64_t bytes, int64_t chunk, int8_t *die_out)
{
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    BSM_GUARD(addr_die_map_host(device, ptr, bytes, chunk, die_out))
}

int bsm_probe_latency(int device, int32_t n_lines, const int64_t *line_off, int32_t reps, float *lat_out,
                      int32_t *seen_out)
{
    if (n_lines <= 0 || !line_off || !lat_out || !seen_out)
        return BSM_ERR_INVALID_ARG;
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    try {
        std::vector<int64_t> lines(line_off, line_off + n_lines);
        std::vector<float> lat;
        std::vector<int32_t> seen;
        int rc = probe_latency_host(device, lines, reps, lat, seen);
        if (rc)
            return rc;
        std::memcpy(lat_out, lat.data(), sizeof(float) * lat.size());
        std::memcpy(seen_out, seen.data(), sizeof(int32_t) * seen.size());
        return BSM_OK;
    } catch (const std::bad_alloc &) {
        return BSM_ERR_NOMEM;
    }
}

int bsm_schedule_host(const bsm_schedule_desc *d, bsm_schedule_out *out) { BSM_GUARD(schedule_host(d, out)) }

int bsm_device_status(int device, uint32_t *status_out)
{
    if (!status_out)
        return BSM_ERR_INVALID_ARG;
    if (device < 0 && cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    int count = 0;
    if (cudaGetDeviceCount(&count) != cudaSuccess || device >= count || device >= kMaxDevices)
        return BSM_ERR_NO_DEVICE;
    if (cudaError_t e = cudaDeviceSynchronize())
        return cuda_error(e, "cudaDeviceSynchronize");
    // the library's word exists once a plan or probe initialised the device;
    // reading it allocates nothing (a caller of bsm_softmax_noalloc alone
    // has only the fixed array's words)
    uint32_t *word = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_mu);
        if (g_dev[device].ready)
            word = g_dev[device].status;
    }
    uint32_t bits = 0;
    if (word) {
        if (cudaError_t e = cudaMemcpy(&bits, word, sizeof(uint32_t), cudaMemcpyDeviceToHost))
            return cuda_error(e, "cudaMemcpy(status)");
    }
    uint32_t na = 0;
    if (int rc = noalloc_status(device, &na, 0))
        return rc;
    *status_out = bits | na;
    return BSM_OK;
}

int bsm_device_status_clear(int device)
{
    DeviceCtx *c = nullptr;
    int rc = device_ctx(device, &c);
    if (rc)
        return rc;
    if (device < 0)
        cudaGetDevice(&device);
    if (cudaError_t e = cudaDeviceSynchronize())
        return cuda_error(e, "cudaDeviceSynchronize");
    if (cudaError_t e = cudaMemset(c->status, 0, 8 * sizeof(uint32_t)))
        return cuda_error(e, "cudaMemset(status)");
    uint32_t na = 0;
    if ((rc = noalloc_status(device, &na, 1)))
        return rc;
    if (cudaError_t e = cudaDeviceSynchronize())
        return cuda_error(e, "cudaDeviceSynchronize");
    return BSM_OK;
}

int bsm_device_debug(int device, uint32_t out[8])
{
    if (!out)
        return BSM_ERR_INVALID_ARG;
    DeviceCtx *c = nullptr;
    int rc = device_ctx(device, &c);
    if (rc)
        return rc;
    if (cudaError_t e = cudaDeviceSynchronize())
        return cuda_error(e, "cudaDeviceSynchronize");
    if (cudaError_t e = cudaMemcpy(out, c->status, 8 * sizeof(uint32_t), cudaMemcpyDeviceToHost))
        return cuda_error(e, "cudaMemcpy(status)");
    return BSM_OK;
}

void bsm_set_device_checks(int on) { g_checked.store(on ? 1 : 0); }

const char *bsm_last_cuda_error(void) { return t_last_error.c_str(); }

int64_t bsm_ragged_extent(int64_t n, const int64_t *offsets, const int32_t *rows, const int32_t *cols)
{
    if (n < 0 || (n > 0 && (!offsets || !rows || !cols)))
        return -1;
    int64_t end = 0;
    for (int64_t s = 0; s < n; ++s) {
        if (rows[s] <= 0)
            continue;
        if (offsets[s] < 0 || cols[s] < 0)
            return -1;
        const int64_t span = int64_t(rows[s]) * cols[s];     // < 2^62
        if (offsets[s] > INT64_MAX - span)
            return -1;
        end = std::max<int64_t>(end, offsets[s] + span);
    }
    return end;
}

int64_t bsm_max_row_bytes(int device)
{
    DeviceCtx *c = nullptr;
    if (device_ctx(device, &c))
        return 0;
    return max_row_bytes_for(*c);
}

const char *bsm_status_string(int status)
{
    switch (status) {
    case BSM_OK:
        return "ok";
    case BSM_ERR_INVALID_ARG:
        return "invalid argument";
    case BSM_ERR_MISALIGNED:
        return "misaligned: pointers, slice offsets and row lengths must be multiples of 16 bytes";
    case BSM_ERR_UNSUPPORTED:
        return "unsupported: shape outside the kernel's limits, or too many patches";
    case BSM_ERR_CUDA:
        return "CUDA runtime error";
    case BSM_ERR_DEVICE_BOUNDS:
        return "a kernel met a patch outside the buffers";
    case BSM_ERR_TIMEOUT:
        return "a kernel wait ran out of time";
    case BSM_ERR_NO_DEVICE:
        return "no usable CUDA device";
    case BSM_ERR_NOMEM:
        return "out of memory";
    case BSM_ERR_TOO_LARGE:
        return "batch needs more patches than bsm_softmax_noalloc's fixed scratch holds "
               "(BSM_NOALLOC_MAX_PATCHES)";
    default:
        return "unknown status";
    }
}

int bsm_version(void) { return (1 << 16) | 0; }

}  // extern "C"
