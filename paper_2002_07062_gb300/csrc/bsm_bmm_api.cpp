// bsm_bmm_api.cpp -- C ABI of the batched matrix product (bsm_bmm): argument
// checks, output tiles as patches under the slice scheduler's policies, TMA
// tensor maps, a small plan cache.

#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <list>
#include <mutex>
#include <new>
#include <numeric>
#include <vector>

#include "bsm_internal.h"
#include "bsm_trace.h"

namespace bsm {

int topology_get(int device, int force, bsm_topology *out);
int device_status_word(int device, uint32_t **out);

namespace {

using EncodeTiled = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                 const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                 CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

struct GemmDev {
    bool ready = false;
    int n_sm = 0, smem_optin = 0;
    uint32_t *status = nullptr;
};

std::mutex g_gemm_mu;
GemmDev g_gdev[64];
EncodeTiled g_encode = nullptr;

int gemm_device(int device, GemmDev **out)
{
    if (device < 0 || device >= 64)
        return BSM_ERR_NO_DEVICE;
    GemmDev &d = g_gdev[device];
    if (!d.ready) {
        if (cudaDeviceGetAttribute(&d.n_sm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, device) != cudaSuccess)
            return BSM_ERR_NO_DEVICE;
        if (int e = gemm_set_smem_limit(d.smem_optin))
            return record_cuda_error(e, "cudaFuncSetAttribute(bmm)");
        if (!g_encode) {
            void *fn = nullptr;
            cudaDriverEntryPointQueryResult q{};
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) !=
                    cudaSuccess ||
                !fn)
                return BSM_ERR_NO_DEVICE;
            g_encode = reinterpret_cast<EncodeTiled>(fn);
        }
        if (int rc = device_status_word(device, &d.status))
            return rc;
        d.ready = true;
    }
    *out = &d;
    return BSM_OK;
}

// Operand view of a (rows_total x K) bf16 row-major matrix as K/64 blocks of
// 64 columns: dims (64, rows, K/64), one box = box_rows rows x kbs blocks,
// 128-byte swizzle; in shared memory the blocks follow one another, each
// box_rows x 128 bytes -- the K-major layout the MMA descriptors read.
int make_operand_map(CUtensorMap *m, const void *base, int64_t rows_total, int64_t K, int box_rows, int kbs)
{
    const cuuint64_t dims[3] = {64u, static_cast<cuuint64_t>(rows_total), static_cast<cuuint64_t>(K / 64)};
    const cuuint64_t strides[2] = {static_cast<cuuint64_t>(K * 2), 128u};
    const cuuint32_t box[3] = {64u, static_cast<cuuint32_t>(box_rows), static_cast<cuuint32_t>(kbs)};
    const cuuint32_t estr[3] = {1u, 1u, 1u};
    const CUresult r = g_encode(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? BSM_OK : BSM_ERR_INVALID_ARG;
}

// box_rows x (128 bytes) boxes of a (rows_total x cols) row-major matrix, 128-byte swizzle
int make_map(CUtensorMap *m, const void *base, int64_t rows_total, int64_t cols, int box_rows, bool f32 = false)
{
    const int es = f32 ? 4 : 2;
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(cols), static_cast<cuuint64_t>(rows_total)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(cols * es)};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(128 / es), static_cast<cuuint32_t>(box_rows)};
    const cuuint32_t estr[2] = {1u, 1u};
    const CUresult r = g_encode(m, f32 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                                const_cast<void *>(base), dims, strides, box,
                                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? BSM_OK : BSM_ERR_INVALID_ARG;
}

struct GemmPlan {
    int device = 0, policy = 0, bn = 0, grid = 0;
    int want_stages = 0, want_bufs = 0, want_kbs = 0;   // caller's choices (0 = automatic)
    bool out_bf16 = false;
    const void *a = nullptr, *bt = nullptr;
    void *c = nullptr;
    int64_t B = 0, M = 0, N = 0, K = 0;
    CUtensorMap ta{}, tb{}, tc{};
    GemmArgs args{};
    std::vector<int32_t> whole_begin;   // WHOLE_GPU: first tile of each slice
    cudaGraphExec_t whole_graph = nullptr;   // WHOLE_GPU: the per-slice launches as one graph
    void *blob = nullptr;
};

std::list<GemmPlan *> g_gcache;

void free_plan(GemmPlan *p)
{
    if (p) {
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
}

// WHOLE_GPU: one launch per slice, one after another (Sec. 3), a
// launch-bound loop; captured once as a CUDA graph when the batch has at
// most this many slices (null if the capture fails: kernel-by-kernel launches)
constexpr int64_t kMaxGraphLaunches = 4096;

cudaGraphExec_t capture_whole_gpu(const GemmPlan *p)
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
        GemmArgs a = p->args;
        for (int64_t s = 0; s < p->B; ++s) {
            a.item_begin = p->whole_begin[s];
            a.item_end = p->whole_begin[s + 1];
            if (launch_bmm(&p->ta, &p->tb, &p->tc, a, p->bn, p->out_bf16, p->grid, st)) {
                ok = false;
                break;
            }
        }
        const cudaError_t ec = cudaStreamEndCapture(st, &g);
        ok = ok && ec == cudaSuccess && g != nullptr;
    }
    if (ok && cudaGraphInstantiate(&e, g, 0) != cudaSuccess)
        e = nullptr;
    if (g)
        cudaGraphDestroy(g);
    cudaStreamDestroy(st);
    cudaGetLastError();
    return e;
}

int build_plan(GemmPlan *p, const GemmDev &dev)
{
    TraceRange trace("bsm_bmm_plan_create");
    const int bn = p->bn;
    const int64_t mt = p->M / 128, nt = p->N / bn;
    const int64_t n_items = p->B * mt * nt;
    if (n_items > INT32_MAX)
        return BSM_ERR_UNSUPPORTED;
    std::vector<GemmItem> items(static_cast<size_t>(n_items));
    std::vector<int32_t> slice_first(static_cast<size_t>(p->B + 1));
    int64_t k = 0;
    for (int64_t s = 0; s < p->B; ++s) {
        slice_first[s] = static_cast<int32_t>(k);
        for (int64_t i = 0; i < mt; ++i)
            for (int64_t j = 0; j < nt; ++j)
                items[k++] = GemmItem{static_cast<int32_t>(s), static_cast<int32_t>(i * 128),
                                      static_cast<int32_t>(j * bn), 0};
    }
    slice_first[p->B] = static_cast<int32_t>(k);

    int n_queues = 1;
    int32_t qbeg[BSM_MAX_DIES] = {0}, qlen[BSM_MAX_DIES] = {0};
    int8_t sm_die[BSM_MAX_SM];
    std::memset(sm_die, 0, sizeof sm_die);
    bool use_die = false;
    int steal = 0;
    qlen[0] = static_cast<int32_t>(n_items);
    if (p->policy == BSM_POLICY_CBMF || p->policy == BSM_POLICY_CBMF_LB || p->policy == BSM_POLICY_MINIMAX) {
        bsm_topology topo;
        if (int rc = topology_get(p->device, 0, &topo))
            return rc;
        if (topo.separable && n_items > 0) {
            // patch bytes: the tile's rows of A (contiguous) -- the operand it streams most
            const int64_t abytes = p->B * p->M * p->K * 2;
            int64_t chunk = std::max<int64_t>(128, (topo.granularity + 127) & ~int64_t(127));
            while ((abytes + chunk - 1) / chunk > (1ll << 24))
                chunk *= 2;
            const int64_t nch = (abytes + chunk - 1) / chunk;
            std::vector<int8_t> amap(static_cast<size_t>(nch));
            if (int rc = addr_die_map_host(p->device, p->a, abytes, chunk, amap.data()))
                return rc;
            std::vector<int64_t> pb(items.size()), pe(items.size()), cost(items.size());
            for (size_t i = 0; i < items.size(); ++i) {
                pb[i] = ((int64_t)items[i].slice * p->M + items[i].m0) * p->K * 2;
                pe[i] = pb[i] + 128 * p->K * 2;
                cost[i] = pe[i] - pb[i] + (int64_t)bn * p->K * 2 + 128ll * bn * (p->out_bf16 ? 2 : 4);
            }
            int32_t units[BSM_MAX_DIES] = {std::max(1, topo.sm_per_die[0]), std::max(1, topo.sm_per_die[1])};
            bsm_schedule_desc sd{};
            sd.n_banks = 2;
            sd.n_patches = n_items;
            sd.patch_begin = pb.data();
            sd.patch_end = pe.data();
            sd.n_maps = 1;
            sd.chunk[0] = chunk;
            sd.n_chunks[0] = nch;
            sd.bank_of_chunk[0] = amap.data();
            sd.tie_seed = 0x2002070600ull;
            sd.balance = p->policy == BSM_POLICY_CBMF_LB;
            sd.method = p->policy == BSM_POLICY_MINIMAX;
            sd.units = units;
            sd.l_near = std::max<int64_t>(1, std::llround(topo.l_near));
            sd.l_far = std::max<int64_t>(1, std::llround(topo.l_far));
            sd.cost = cost.data();
            std::vector<int64_t> bob(items.size() * 2);
            std::vector<uint8_t> ov(items.size());
            std::vector<int32_t> bank(items.size()), qi(items.size()), moved(items.size());
            int64_t N[BSM_MAX_DIES] = {0}, L[BSM_MAX_DIES] = {0}, ql[BSM_MAX_DIES] = {0}, wb[4] = {0}, wa[4] = {0};
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
            if (int rc = schedule_host(&sd, &so))
                return rc;
            std::vector<GemmItem> ordered(items.size());
            for (size_t i = 0; i < items.size(); ++i)
                ordered[i] = items[static_cast<size_t>(qi[i])];
            items.swap(ordered);
            n_queues = 2;
            qbeg[0] = 0;
            qlen[0] = static_cast<int32_t>(ql[0]);
            qbeg[1] = qlen[0];
            qlen[1] = static_cast<int32_t>(ql[1]);
            std::memcpy(sm_die, topo.sm_die, sizeof sm_die);
            for (int s = 0; s < BSM_MAX_SM; ++s)
                if (sm_die[s] < 0)
                    sm_die[s] = 0;
            use_die = true;
            steal = p->policy != BSM_POLICY_CBMF;
        }
    }

    auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
    const size_t items_b = sizeof(GemmItem) * items.size(), slices_b = sizeof(int32_t) * slice_first.size();
    const size_t o_items = 0, o_slices = up(items_b), o_smdie = o_slices + up(slices_b), o_heads = o_smdie + 256,
                 blob_b = o_heads + 256;
    std::vector<unsigned char> host(blob_b, 0);
    if (items_b)
        std::memcpy(&host[o_items], items.data(), items_b);
    std::memcpy(&host[o_slices], slice_first.data(), slices_b);
    std::memcpy(&host[o_smdie], sm_die, sizeof sm_die);
    if (cudaMalloc(&p->blob, blob_b) != cudaSuccess)
        return BSM_ERR_NOMEM;
    if (cudaError_t e = cudaMemcpy(p->blob, host.data(), blob_b, cudaMemcpyHostToDevice))
        return record_cuda_error(static_cast<int>(e), "cudaMemcpy(bmm plan)");
    unsigned char *b = static_cast<unsigned char *>(p->blob);

    GemmArgs &a = p->args;
    a.c = p->c;
    a.B = static_cast<int32_t>(p->B);
    a.M = static_cast<int32_t>(p->M);
    a.N = static_cast<int32_t>(p->N);
    a.K = static_cast<int32_t>(p->K);
    a.items = reinterpret_cast<const GemmItem *>(b + o_items);
    a.n_items = static_cast<int32_t>(n_items);
    a.slice_first_item = reinterpret_cast<const int32_t *>(b + o_slices);
    a.n_slices = static_cast<int32_t>(p->B);
    a.n_queues = n_queues;
    for (int q = 0; q < BSM_MAX_DIES; ++q) {
        a.queue_begin[q] = qbeg[q];
        a.queue_len[q] = qlen[q];
    }
    a.steal = steal;
    a.heads = reinterpret_cast<uint32_t *>(b + o_heads);
    a.sm_die = use_die ? reinterpret_cast<const int8_t *>(b + o_smdie) : nullptr;
    // shared memory split: with few K blocks per tile the output dominates,
    // so favour store buffers; with many, favour stages in flight
    // and fetch several K blocks per copy when the tile has them (longer
    // runs of each operand row per request), keeping two stages or more
    const int64_t kb = p->K / 64;
    int kbs = p->want_kbs;
    if (!kbs) {
        kbs = 1;
        for (int g : {4, 2})
            if (kb % g == 0 &&
                (dev.smem_optin - gemm_fixed_smem(bn, p->out_bf16, 2)) / (g * gemm_stage_bytes(bn)) >= 2) {
                kbs = g;
                break;
            }
    }
    if (kb % kbs)
        return BSM_ERR_UNSUPPORTED;
    int bufs = p->want_bufs ? p->want_bufs : (kb <= 2 ? 4 : 2);
    int fit = 0;
    for (;; --bufs) {
        fit = (dev.smem_optin - gemm_fixed_smem(bn, p->out_bf16, bufs)) / (kbs * gemm_stage_bytes(bn));
        if (fit >= 2 || bufs <= 2 || p->want_bufs)
            break;
    }
    // an output-heavy tile left with two stages: a third stage beats the
    // extra store buffers (E1, 384 x (512x64)(64x512): 3 stages x 2 buffers
    // 41.60 us against 2 x 4 41.85 us, same box)
    if (!p->want_bufs && !p->want_stages && fit == 2 && bufs > 2) {
        const int fit2 = (dev.smem_optin - gemm_fixed_smem(bn, p->out_bf16, 2)) / (kbs * gemm_stage_bytes(bn));
        if (fit2 >= 3) {
            bufs = 2;
            fit = fit2;
        }
    }
    a.epi_bufs = bufs;
    a.kbs = kbs;
    a.identity = use_die ? 0 : 1;
    a.tiles_m = static_cast<int32_t>(mt);
    a.tiles_n = static_cast<int32_t>(nt);
    a.n_stages = std::min(8, fit);
    if (p->want_stages)
        a.n_stages = p->want_stages <= fit ? p->want_stages : 0;
    a.status = dev.status;
    if (a.n_stages < 2)
        return BSM_ERR_UNSUPPORTED;
    switch (p->policy) {
    case BSM_POLICY_WHOLE_GPU:
        a.mode = PULL_STATIC;
        p->whole_begin = slice_first;
        p->grid = static_cast<int>(std::min<int64_t>(dev.n_sm, mt * nt));
        break;
    case BSM_POLICY_RR:
        a.mode = PULL_RR_SLICE;
        p->grid = static_cast<int>(std::min<int64_t>(dev.n_sm, p->B));
        break;
    default:
        a.mode = PULL_QUEUE;
        p->grid = dev.n_sm;
        break;
    }
    if (int rc = make_operand_map(&p->ta, p->a, p->B * p->M, p->K, 128, kbs))
        return rc;
    if (int rc = make_operand_map(&p->tb, p->bt, p->B * p->N, p->K, bn, kbs))
        return rc;
    if (int rc = make_map(&p->tc, p->c, p->B * p->M, p->N, 32, !p->out_bf16))
        return rc;
    return BSM_OK;
}

int run_plan(GemmPlan *p, bsm_stream_t stream)
{
    TraceRange trace("bsm_bmm_execute");
    int err = 0;
    if (p->policy == BSM_POLICY_WHOLE_GPU && p->whole_graph) {
        err = static_cast<int>(cudaGraphLaunch(p->whole_graph, static_cast<cudaStream_t>(stream)));
    } else if (p->policy == BSM_POLICY_WHOLE_GPU) {
        GemmArgs a = p->args;
        for (int64_t s = 0; s < p->B; ++s) {
            a.item_begin = p->whole_begin[s];
            a.item_end = p->whole_begin[s + 1];
            if ((err = launch_bmm(&p->ta, &p->tb, &p->tc, a, p->bn, p->out_bf16, p->grid, stream)))
                break;
        }
    } else {
        err = launch_bmm(&p->ta, &p->tb, &p->tc, p->args, p->bn, p->out_bf16, p->grid, stream);
    }
    return err ? record_cuda_error(err, "bmm kernel launch") : BSM_OK;
}

int bmm_impl(const void *a, const void *bt, void *c, int64_t B, int64_t M, int64_t N, int64_t K, int out_dtype,
             int policy, int n_stages, int epi_bufs, int kbs, bsm_stream_t stream)
{
    if (B < 0 || M < 0 || N < 0 || K < 0 || (out_dtype != BSM_F32 && out_dtype != BSM_BF16) ||
        policy < BSM_POLICY_WHOLE_GPU || policy > BSM_POLICY_MINIMAX || n_stages < 0 || n_stages == 1 ||
        n_stages > 8 || epi_bufs < 0 || epi_bufs == 1 || epi_bufs > 4 || (kbs != 0 && kbs != 1 && kbs != 2 &&
                                                                           kbs != 4))
        return BSM_ERR_INVALID_ARG;
    if (B == 0 || M == 0 || N == 0)
        return BSM_OK;
    if (K == 0 || M % 128 || N % 64 || K % 64)
        return BSM_ERR_UNSUPPORTED;
    if (M > (1 << 24) || N > (1 << 24) || K > (1 << 24) || B > (int64_t(1) << 31) / std::max(M, N))
        return BSM_ERR_UNSUPPORTED;
    if (!a || !bt || !c)
        return BSM_ERR_INVALID_ARG;
    const uintptr_t ca = reinterpret_cast<uintptr_t>(c);
    if ((reinterpret_cast<uintptr_t>(a) & 15) || (reinterpret_cast<uintptr_t>(bt) & 15) || (ca & 15))
        return BSM_ERR_MISALIGNED;
    const uintptr_t clen = static_cast<uintptr_t>(B * M * N * (out_dtype == BSM_BF16 ? 2 : 4));
    const uintptr_t alen = static_cast<uintptr_t>(B * M * K * 2), blen = static_cast<uintptr_t>(B * N * K * 2);
    auto overlap = [](uintptr_t x, uintptr_t xl, uintptr_t y, uintptr_t yl) { return x < y + yl && y < x + xl; };
    if (overlap(ca, clen, reinterpret_cast<uintptr_t>(a), alen) ||
        overlap(ca, clen, reinterpret_cast<uintptr_t>(bt), blen))
        return BSM_ERR_INVALID_ARG;
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    std::lock_guard<std::mutex> lk(g_gemm_mu);
    GemmDev *dev = nullptr;
    if (int rc = gemm_device(device, &dev))
        return rc;
    for (auto it = g_gcache.begin(); it != g_gcache.end(); ++it) {
        GemmPlan *p = *it;
        if (p->device == device && p->a == a && p->bt == bt && p->c == c && p->B == B && p->M == M && p->N == N &&
            p->K == K && p->out_bf16 == (out_dtype == BSM_BF16) && p->policy == policy &&
            p->want_stages == n_stages && p->want_bufs == epi_bufs && p->want_kbs == kbs) {
            g_gcache.splice(g_gcache.begin(), g_gcache, it);
            return run_plan(p, stream);
        }
    }
    GemmPlan *p = new GemmPlan();
    p->device = device;
    p->policy = policy;
    p->want_stages = n_stages;
    p->want_bufs = epi_bufs;
    p->want_kbs = kbs;
    p->bn = N % 256 == 0 ? 256 : (N % 128 == 0 ? 128 : 64);
    p->out_bf16 = out_dtype == BSM_BF16;
    p->a = a;
    p->bt = bt;
    p->c = c;
    p->B = B;
    p->M = M;
    p->N = N;
    p->K = K;
    if (int rc = build_plan(p, *dev)) {
        free_plan(p);
        return rc;
    }
    if (p->policy == BSM_POLICY_WHOLE_GPU && p->B > 0 && p->B <= kMaxGraphLaunches)
        p->whole_graph = capture_whole_gpu(p);
    g_gcache.push_front(p);
    while (g_gcache.size() > 16) {
        free_plan(g_gcache.back());
        g_gcache.pop_back();
    }
    return run_plan(p, stream);
}

}  // namespace
}  // namespace bsm

extern "C" int bsm_bmm(const void *a, const void *bt, void *c, int64_t B, int64_t M, int64_t N, int64_t K,
                       int out_dtype, int policy, bsm_stream_t stream)
{
    try {
        return bsm::bmm_impl(a, bt, c, B, M, N, K, out_dtype, policy, 0, 0, 0, stream);
    } catch (const std::bad_alloc &) {
        return BSM_ERR_NOMEM;
    }
}

extern "C" int bsm_bmm_ex(const void *a, const void *bt, void *c, int64_t B, int64_t M, int64_t N, int64_t K,
                          int out_dtype, int policy, int n_stages, int epi_bufs, int k_blocks_per_stage,
                          bsm_stream_t stream)
{
    try {
        return bsm::bmm_impl(a, bt, c, B, M, N, K, out_dtype, policy, n_stages, epi_bufs, k_blocks_per_stage,
                             stream);
    } catch (const std::bad_alloc &) {
        return BSM_ERR_NOMEM;
    }
}
