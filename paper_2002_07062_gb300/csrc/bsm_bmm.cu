// bsm_bmm.cu -- the paper's second batch algorithm (Sec. 6: batch 384 of
// (512 x 64) x (64 x 512) and of (512 x 512) x (512 x 64)): the batched
// matrix product C_s = A_s * Bt_s^T, on the 5th-generation tensor cores.
//
// One persistent CTA per SM, 10 warps:
//   warp 0, lane 0  producer: pulls output tiles (BM x BN of one slice) from
//                   the schedule (the slice scheduler's policies), streams the
//                   tile's A rows and Bt rows, 64 columns of K at a time, into
//                   a ring of shared-memory stages with 2-D TMA copies
//                   (128-byte swizzle, completion on the stage's mbarrier);
//   warp 1          owns the tensor memory (allocates two BN-column fp32
//                   accumulators, frees them at the end); its lane 0 issues
//                   tcgen05.mma (M = 128, N = BN, K = 16 per instruction) from
//                   shared-memory descriptors and commits each stage back to
//                   the producer and each finished tile to the epilogue;
//   warps 2-9       epilogue: tcgen05.ld of the accumulator (one TMEM lane =
//                   one output row per thread), round, write 32 rows x 128
//                   bytes at a time into a 128-byte-swizzled shared buffer
//                   (conflict-free), and one lane stores it with a 2-D TMA
//                   tensor store; two buffers per warp, so the next unit is
//                   converted while the last one drains.
// The accumulators are double-buffered so the epilogue of a tile overlaps the
// MMAs of the next.  Every wait is bounded (2 s of %globaltimer): on expiry
// the CTA records BSM_DEV_TIMEOUT and leaves; the tensor memory is always
// deallocated before the CTA exits.

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "bsm_internal.h"

namespace bsm {
namespace {

constexpr int kBM = 128;
constexpr int kBK = 64;                 // bf16 columns per stage: one 128-byte swizzle row
constexpr int kEpiWarps = 8;
constexpr int kGemmThreads = (2 + kEpiWarps) * 32;
constexpr int kEpiBuf = 32 * 128;       // one store unit: 32 rows x 128 bytes

// Epilogue warps with work: two per TMEM lane quarter when a tile row block
// has at least two 128-byte store units, else one.
__host__ __device__ constexpr int epi_active(int bn, bool out_bf16)
{
    return (bn * (out_bf16 ? 2 : 4)) / 128 >= 2 ? 8 : 4;
}
constexpr int kGemmMaxStages = 8;
constexpr uint64_t kGemmWaitNs = 2000000000ull;

enum : int32_t { GK_DATA = 0, GK_DONE = 2 };

struct GemmMeta {
    int32_t slice, m0, n0, kind;
};

struct GemmSmem {
    uint64_t full[kGemmMaxStages];
    uint64_t empty[kGemmMaxStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    GemmMeta smeta[kGemmMaxStages];
    GemmMeta tmeta[2];
    uint32_t tmem_base;
    int32_t abort_flag;
};
static_assert(sizeof(GemmSmem) <= 1024, "gemm header");

__device__ __forceinline__ uint32_t saddr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t gtimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t gemm_smid()
{
    uint32_t s;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(s));
    return s;
}

__device__ __forceinline__ void bar_init(uint64_t *b, uint32_t n)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(saddr(b)), "r"(n) : "memory");
}

__device__ __forceinline__ void bar_arrive(uint64_t *b)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(saddr(b)) : "memory");
}

__device__ __forceinline__ void bar_expect(uint64_t *b, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(saddr(b)), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ bool bar_try(uint64_t *b, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(saddr(b)), "r"(parity), "r"(50000u)
        : "memory");
    return ok != 0;
}

// Bounded wait for the phase of `parity`; false on abort or time out.
__device__ __noinline__ bool bar_wait(uint64_t *b, uint32_t parity, const volatile int32_t *abort)
{
    if (bar_try(b, parity))
        return true;
    const uint64_t t0 = gtimer();
    for (uint32_t it = 0; it < (1u << 28); ++it) {
        if (bar_try(b, parity))
            return true;
        if (abort && *abort)
            return false;
        if (gtimer() - t0 > kGemmWaitNs)
            return false;
    }
    return false;
}

// 3-D TMA tile load: box at (c0 = column in the K block, c1 = row, c2 = K block).
__device__ __forceinline__ void tma_load_3d(void *dst, const CUtensorMap *map, int32_t c0, int32_t c1, int32_t c2,
                                            uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, "
        "%3, %4}], [%5];" ::"r"(saddr(dst)),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(c0), "r"(c1), "r"(c2), "r"(saddr(bar))
        : "memory");
}

// Tile record of queue entry idx: read from the plan, or computed when the
// plan keeps tiles in their natural order (slice, row block, column block).
template <int BN> __device__ __forceinline__ GemmItem tile_at(const GemmArgs &a, int32_t idx)
{
    if (idx < 0 || idx >= a.n_items)
        return GemmItem{-1, 0, 0, 0};
    if (!a.identity)
        return a.items[idx];
    const int32_t per = a.tiles_m * a.tiles_n;
    const int32_t s = idx / per, r = idx - s * per;
    return GemmItem{s, (r / a.tiles_n) * 128, (r % a.tiles_n) * BN, 0};
}

// Shared-memory matrix descriptor of a K-major operand tile whose rows are
// 128 bytes (64 bf16) laid out with the 128-byte swizzle by TMA: start
// address (16-byte units), leading-dimension offset (unused for this
// layout: 1), stride between 8-row groups = 1024 bytes, descriptor version 1,
// base offset 0 (tiles are 1024-byte aligned), swizzle mode 2 = 128 bytes.
__device__ __forceinline__ uint64_t smem_desc(const void *tile)
{
    const uint64_t a = (saddr(tile) & 0x3FFFFu) >> 4;
    return a | (1ull << 16) | (uint64_t(1024 >> 4) << 32) | (1ull << 46) | (2ull << 61);
}

// Instruction descriptor of kind::f16: fp32 accumulator, bf16 A and B, both
// K-major, N = BN, M = 128.
template <int BN> __device__ __forceinline__ uint32_t mma_idesc()
{
    return (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(BN >> 3) << 17) | (uint32_t(kBM >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on `bar` when every tcgen05.mma issued so far by this thread is done.
__device__ __forceinline__ void mma_commit(uint64_t *bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(saddr(bar))
                 : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

// 32 consecutive fp32 columns of this thread's TMEM lane (no wait).
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, uint32_t *r)
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, "
        "%14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 2-D TMA tensor store of a shared-memory box at (c0 = column, c1 = row).
__device__ __forceinline__ void tma_store_2d(const CUtensorMap *map, int32_t c0, int32_t c1, const void *src)
{
    asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%1, %2}], [%3];" ::"l"(
                     reinterpret_cast<uint64_t>(map)),
                 "r"(c0), "r"(c1), "r"(saddr(src))
                 : "memory");
    asm volatile("cp.async.bulk.commit_group;" ::: "memory");
}

__device__ __forceinline__ void st_shared_v4(uint32_t addr, uint32_t x, uint32_t y, uint32_t z, uint32_t w)
{
    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(x), "r"(y), "r"(z), "r"(w)
                 : "memory");
}

// Programmatic dependent launch: the kernel may start while the previous
// kernel of the stream is finishing; this waits until that kernel has
// completed and its writes are visible (a no-op without such a predecessor).
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
// Let the next kernel of the stream start its launch (it still waits on its own
// grid_dependency_wait before touching memory).
__device__ __forceinline__ void grid_launch_dependents() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

__device__ __forceinline__ uint32_t bf16x2(float lo, float hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// The next tiles of this CTA under the plan's policy (same modes as the
// softmax kernel: static list, whole slices round robin, die queues).
struct GemmPuller {
    const GemmArgs &a;
    int32_t k = 0, slice = -1, cur = 0, end = 0, q = 0, die = 0;
    bool first = true;

    __device__ explicit GemmPuller(const GemmArgs &args) : a(args)
    {
        if (a.mode == PULL_QUEUE && a.sm_die) {
            const int d = a.sm_die[gemm_smid() & (BSM_MAX_SM - 1)];
            die = (d >= 0 && d < a.n_queues) ? d : 0;
        }
        if (a.mode == PULL_RR_SLICE)
            slice = static_cast<int32_t>(blockIdx.x) - static_cast<int32_t>(gridDim.x);
    }

    __device__ int32_t next()
    {
        if (a.mode == PULL_STATIC) {
            const int64_t idx = (int64_t)a.item_begin + blockIdx.x + (int64_t)k * gridDim.x;
            ++k;
            return idx < a.item_end ? static_cast<int32_t>(idx) : -1;
        }
        if (a.mode == PULL_RR_SLICE) {
            while (cur >= end) {
                slice += gridDim.x;
                if (slice >= a.n_slices)
                    return -1;
                cur = a.slice_first_item[slice];
                end = a.slice_first_item[slice + 1];
            }
            return cur++;
        }
        if (a.n_queues == 1) {
            // one queue: CTA i starts with tile i without touching the
            // counter; later claims are counter + gridDim.x
            const uint32_t t = first ? blockIdx.x : atomicAdd(&a.heads[0], 1u) + gridDim.x;
            first = false;
            return t < static_cast<uint32_t>(a.queue_len[0]) ? a.queue_begin[0] + static_cast<int32_t>(t) : -1;
        }
        const int tries = a.steal ? a.n_queues : 1;
        while (q < tries) {
            const int qq = (die + q) % a.n_queues;
            const uint32_t t = atomicAdd(&a.heads[qq], 1u);
            if (t < static_cast<uint32_t>(a.queue_len[qq]))
                return a.queue_begin[qq] + static_cast<int32_t>(t);
            ++q;
        }
        return -1;
    }
};

template <int BN, bool kOutBf16>
__global__ void __launch_bounds__(kGemmThreads, 1)
    bmm_persistent(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const GemmArgs a)
{
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    // the 128-byte swizzle wants 1024-byte aligned tiles: align at run time
    // (the launch asks for 1 KiB of slack)
    unsigned char *smem = smem_raw + ((1024u - (saddr(smem_raw) & 1023u)) & 1023u);
    GemmSmem &h = *reinterpret_cast<GemmSmem *>(smem);
    constexpr uint32_t kABytes = kBM * kBK * 2;
    constexpr uint32_t kBBytes = BN * kBK * 2;
    const int G = a.kbs;                                   // K blocks per stage (one 3-D copy each)
    const uint32_t stage_bytes = static_cast<uint32_t>(G) * (kABytes + kBBytes);
    constexpr uint32_t kTmemCols = 2 * BN;
    constexpr int kActive = epi_active(BN, kOutBf16);
    const int bufs = a.epi_bufs;                           // store buffers per active warp
    unsigned char *epi = smem + 1024;
    unsigned char *stages = smem + 1024 + kActive * bufs * kEpiBuf;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = a.n_stages;
    const int NS = a.K / (kBK * G);                        // stages per tile

    if (warp == 0) {
        // ------------------------------------------------------- producer
        // The first claim and the tensor-map fetches are issued before the
        // barriers are set up; the producer streams as soon as they exist,
        // without waiting for the tensor-memory allocation.
        GemmPuller pull(a);
        int32_t idx = -1;
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmA)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmB)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmC)) : "memory");
            const bool static_first = a.mode != PULL_QUEUE || a.n_queues == 1;
            if (static_first)
                idx = pull.next();                 // no memory access: before the wait
            for (int s = 0; s < S; ++s) {
                bar_init(&h.full[s], 1);
                bar_init(&h.empty[s], 1);
            }
            for (int b = 0; b < 2; ++b) {
                bar_init(&h.tfull[b], 1);
                bar_init(&h.tempty[b], kActive);
            }
            bar_init(&h.drain, 1);
            h.abort_flag = 0;
            asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
            // launched early behind the previous kernel of the stream: from
            // here on memory is touched, so wait until that kernel is done
            grid_dependency_wait();
            if (!static_first)
                idx = pull.next();
        }
        __syncwarp();
        asm volatile("barrier.cta.arrive 1, %0;" ::"r"(kGemmThreads) : "memory");   // barriers ready
        grid_launch_dependents();
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            // the next tile is claimed (and its record fetched) while the
            // current one streams, so the ring never waits on the queue
            GemmItem item = tile_at<BN>(a, idx);
            for (;;) {
                const int32_t nidx = idx >= 0 ? pull.next() : -1;
                const bool have = idx >= 0 && idx < a.n_items;
                const bool valid = have && item.slice >= 0 && item.slice < a.B && item.m0 >= 0 &&
                                   item.m0 + kBM <= a.M && item.n0 >= 0 && item.n0 + BN <= a.N;
                if (idx >= 0 && !valid)
                    atomicOr(a.status, BSM_DEV_BOUNDS);     // skip a bad tile, keep going
                GemmItem nitem{};
                const int nks = idx < 0 ? 1 : (valid ? NS : 0);
                for (int kb = 0; kb < nks; ++kb) {
                    const int s = static_cast<int>(it % S);
                    const uint32_t ph = (it / S) & 1u;
                    if (!bar_wait(&h.empty[s], ph ^ 1u, &h.abort_flag)) {
                        ok = false;
                        break;
                    }
                    ++it;
                    if (idx < 0) {
                        h.smeta[s].kind = GK_DONE;
                        bar_arrive(&h.full[s]);
                        break;
                    }
                    if (kb == 0)
                        h.smeta[s] = GemmMeta{item.slice, item.m0, item.n0, GK_DATA};
                    unsigned char *st = stages + (size_t)s * stage_bytes;
                    bar_expect(&h.full[s], stage_bytes);
                    tma_load_3d(st, &tmA, 0, item.slice * a.M + item.m0, kb * G, &h.full[s]);
                    tma_load_3d(st + G * kABytes, &tmB, 0, item.slice * a.N + item.n0, kb * G, &h.full[s]);
                    if (kb == 0)
                        nitem = tile_at<BN>(a, nidx);
                }
                if (!ok || idx < 0)
                    break;
                if (nks == 0)
                    nitem = tile_at<BN>(a, nidx);
                idx = nidx;
                item = nitem;
            }
            if (!ok) {
                atomicOr(a.status, BSM_DEV_TIMEOUT);
                h.abort_flag = 1;
            }
            // copies still in flight land before the CTA may leave (no-op on
            // the normal path, where the MMA issuer consumed every stage)
            for (uint32_t j = it > static_cast<uint32_t>(S) ? it - S : 0u; j < it; ++j)
                bar_wait(&h.full[j % S], (j / S) & 1u, nullptr);
            if (a.mode == PULL_QUEUE) {
                __threadfence();
                const uint32_t prev = atomicAdd(&a.heads[BSM_MAX_DIES], 1u);
                if (prev == gridDim.x - 1) {
                    for (int d = 0; d < BSM_MAX_DIES; ++d)
                        atomicExch(&a.heads[d], 0u);
                    atomicExch(&a.heads[BSM_MAX_DIES], 0u);
                }
            }
        }
    } else {
        asm volatile("barrier.cta.sync 1, %0;" ::"r"(kGemmThreads) : "memory");          // barriers ready
        if (warp == 1) {
            asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(&h.tmem_base)),
                         "r"(kTmemCols)
                         : "memory");
            asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
        }
        tc_fence_before();
        asm volatile("barrier.cta.sync 2, %0;" ::"r"(kGemmThreads - 32) : "memory");     // TMEM address ready
        tc_fence_after();
        const uint32_t tmem = h.tmem_base;
        if (warp == 1) {
            // ------------------------------------------------------- MMA issuer
            if (lane == 0) {
                // no bounded wait may start before the previous kernel is done
                grid_dependency_wait();
                const uint32_t idesc = mma_idesc<BN>();
                uint32_t it = 0, t = 0;
                bool ok = true;
                for (;;) {
                    int s = static_cast<int>(it % S);
                    uint32_t ph = (it / S) & 1u;
                    if (!bar_wait(&h.full[s], ph, &h.abort_flag)) {
                        ok = false;
                        break;
                    }
                    const GemmMeta m = h.smeta[s];
                    const int buf = static_cast<int>(t & 1u);
                    const uint32_t tph = (t >> 1) & 1u;
                    if (!bar_wait(&h.tempty[buf], tph ^ 1u, &h.abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    h.tmeta[buf] = m;
                    __threadfence_block();              // visible before the MMAs (and their commit)
                    if (m.kind == GK_DONE) {
                        bar_arrive(&h.tfull[buf]);
                        break;
                    }
                    const uint32_t d = tmem + static_cast<uint32_t>(buf * BN);
                    for (int kb = 0; kb < NS; ++kb) {
                        if (kb > 0) {
                            s = static_cast<int>(it % S);
                            ph = (it / S) & 1u;
                            if (!bar_wait(&h.full[s], ph, &h.abort_flag)) {
                                ok = false;
                                break;
                            }
                        }
                        tc_fence_after();
                        unsigned char *st = stages + (size_t)s * stage_bytes;
                        for (int j = 0; j < G; ++j) {
                            const uint64_t ad = smem_desc(st + j * kABytes);
                            const uint64_t bd = smem_desc(st + G * kABytes + j * kBBytes);
    #pragma unroll
                            for (int k = 0; k < kBK / 16; ++k)
                                mma_bf16(d, ad + 2 * k, bd + 2 * k, idesc, (kb | j | k) != 0);
                        }
                        mma_commit(&h.empty[s]);        // the stage is free once these are done
                        ++it;
                    }
                    if (!ok)
                        break;
                    mma_commit(&h.tfull[buf]);          // the accumulator is ready
                    ++t;
                }
                if (!ok) {
                    atomicOr(a.status, BSM_DEV_TIMEOUT);
                    h.abort_flag = 1;
                }
                // every MMA issued has finished before the tensor memory is freed
                mma_commit(&h.drain);
                bar_wait(&h.drain, 0, nullptr);
            }
        } else {
            // ------------------------------------------------------- epilogue
            constexpr int kEs = kOutBf16 ? 2 : 4;
            constexpr int kUnitCols = 128 / kEs;                  // output columns per store unit
            constexpr int kUnits = BN / kUnitCols;                // store units per tile row block
            const int ew = warp - 2;
            const int quarter = warp & 3;                         // TMEM lanes this warp may read
            const int half = ew >> 2;                             // which units of the quarter
            unsigned char *mybuf = epi + ew * bufs * kEpiBuf;
            uint32_t nst = 0;                                     // units stored by this warp
            grid_dependency_wait();                       // before any wait or store
            for (uint32_t t = 0; ew < kActive; ++t) {
                const int buf = static_cast<int>(t & 1u);
                // lane 0 waits; the warp follows its verdict (tcgen05.ld is warp-wide)
                int ok = 0;
                if (lane == 0) {
                    ok = bar_wait(&h.tfull[buf], (t >> 1) & 1u, &h.abort_flag);
                    if (!ok) {
                        atomicOr(a.status, BSM_DEV_TIMEOUT);
                        h.abort_flag = 1;
                    }
                }
                ok = __shfl_sync(0xffffffffu, ok, 0);
                __syncwarp();
                if (!ok)
                    break;
                tc_fence_after();
                const GemmMeta m = h.tmeta[buf];
                if (m.kind == GK_DONE)
                    break;
                const uint32_t tbase =
                    tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(buf * BN);
                const int32_t crow = m.slice * a.M + m.m0 + quarter * 32;
    #pragma unroll 1
                for (int u = half; u < kUnits; u += kActive / 4, ++nst) {
                    uint32_t r[64];
                    tmem_ld32_nowait(tbase + static_cast<uint32_t>(u * kUnitCols), r);
                    if (kOutBf16)
                        tmem_ld32_nowait(tbase + static_cast<uint32_t>(u * kUnitCols + 32), r + 32);
                    tmem_wait_ld();
                    // the buffer about to be rewritten must have been read by its store
                    if (lane == 0) {
                        if (bufs >= 4)
                            asm volatile("cp.async.bulk.wait_group.read 3;" ::: "memory");
                        else if (bufs == 3)
                            asm volatile("cp.async.bulk.wait_group.read 2;" ::: "memory");
                        else
                            asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
                    }
                    __syncwarp();
                    unsigned char *ub = mybuf + (nst % static_cast<uint32_t>(bufs)) * kEpiBuf;
                    const uint32_t sb = saddr(ub) + static_cast<uint32_t>(lane * 128);
    #pragma unroll
                    for (int c = 0; c < 8; ++c) {
                        const uint32_t dst = sb + (static_cast<uint32_t>(c ^ (lane & 7)) << 4);
                        if (kOutBf16) {
                            const float *f = reinterpret_cast<const float *>(r + 8 * c);
                            st_shared_v4(dst, bf16x2(f[0], f[1]), bf16x2(f[2], f[3]), bf16x2(f[4], f[5]),
                                         bf16x2(f[6], f[7]));
                        } else {
                            st_shared_v4(dst, r[4 * c], r[4 * c + 1], r[4 * c + 2], r[4 * c + 3]);
                        }
                    }
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0)
                        tma_store_2d(&tmC, m.n0 + u * kUnitCols, crow, ub);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0)
                    bar_arrive(&h.tempty[buf]);
            }
            // stores complete before the CTA leaves
            if (lane == 0)
                asm volatile("cp.async.bulk.wait_group 0;" ::: "memory");
            __syncwarp();
        }
    }

    // every thread gets here (all waits are bounded); then the owner frees TMEM
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(h.tmem_base), "r"(kTmemCols)
                     : "memory");
    }
}

template <int BN, bool kOutBf16>
int launch_bn(const CUtensorMap &ta, const CUtensorMap &tb, const CUtensorMap &tc, const GemmArgs &a, int grid,
              cudaStream_t st)
{
    const size_t smem = static_cast<size_t>(gemm_fixed_smem(BN, kOutBf16, a.epi_bufs)) +
                        (size_t)a.n_stages * a.kbs * (kBM * kBK * 2 + BN * kBK * 2);
#ifndef BSM_NO_PDL
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kGemmThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return static_cast<int>(cudaLaunchKernelEx(&cfg, bmm_persistent<BN, kOutBf16>, ta, tb, tc, a));
#else
    bmm_persistent<BN, kOutBf16><<<grid, kGemmThreads, smem, st>>>(ta, tb, tc, a);
    return static_cast<int>(cudaGetLastError());
#endif
}

}  // namespace

int gemm_stage_bytes(int bn) { return kBM * kBK * 2 + bn * kBK * 2; }
int gemm_threads() { return kGemmThreads; }
int gemm_fixed_smem(int bn, bool out_bf16, int epi_bufs)
{
    return 2048 + epi_active(bn, out_bf16) * epi_bufs * kEpiBuf;
}

int gemm_set_smem_limit(int bytes)
{
    const void *fns[] = {reinterpret_cast<const void *>(bmm_persistent<64, false>),
                         reinterpret_cast<const void *>(bmm_persistent<64, true>),
                         reinterpret_cast<const void *>(bmm_persistent<128, false>),
                         reinterpret_cast<const void *>(bmm_persistent<128, true>),
                         reinterpret_cast<const void *>(bmm_persistent<256, false>),
                         reinterpret_cast<const void *>(bmm_persistent<256, true>)};
    for (const void *f : fns)
        if (cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes))
            return static_cast<int>(e);
    return 0;
}

int launch_bmm(const void *tmap_a, const void *tmap_b, const void *tmap_c, const GemmArgs &a, int bn,
               bool out_bf16, int grid, void *stream)
{
    const CUtensorMap &ta = *static_cast<const CUtensorMap *>(tmap_a);
    const CUtensorMap &tb = *static_cast<const CUtensorMap *>(tmap_b);
    const CUtensorMap &tc = *static_cast<const CUtensorMap *>(tmap_c);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (bn == 64)
        return out_bf16 ? launch_bn<64, true>(ta, tb, tc, a, grid, st) : launch_bn<64, false>(ta, tb, tc, a, grid, st);
    if (bn == 128)
        return out_bf16 ? launch_bn<128, true>(ta, tb, tc, a, grid, st)
                        : launch_bn<128, false>(ta, tb, tc, a, grid, st);
    return out_bf16 ? launch_bn<256, true>(ta, tb, tc, a, grid, st) : launch_bn<256, false>(ta, tb, tc, a, grid, st);
}

}  // namespace bsm
