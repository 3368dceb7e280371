// bsm_noalloc.cu -- bsm_softmax_noalloc: the batched softmax for callers
// that cannot allocate device memory.
//
// The regular entry points allocate: a plan owns a device table of patches
// and queue counters (cudaMalloc), and the library keeps a status word per
// device.  Some callers cannot allow that -- code running inside a
// pre-sized memory pool or arena (an inference server that has reserved the
// whole device up front, a framework allocator that must see every byte), or
// code that must not add cudaMalloc/cudaFree calls, which synchronise the
// device, to a latency-critical path.  This entry point runs the same
// persistent kernel under the one-queue dynamic schedule (a batch of at most
// one patch per SM dealt statically, as the planned path deals it), with its scratch
// (patch table, queue counters, status words) in one file-scope __device__
// array of fixed size instead of allocated memory.  The caller still passes
// x and y.  Rows must fit one shared-memory stage (BSM_NOALLOC_MAX_ROW_BYTES,
// and the device's own stage limit): the two-pass path of longer rows needs
// per-plan buffers this entry point does not have.
//
// The array is part of the library's device image: every GPU that loads the
// library holds it (about 1.5 MiB) until the process exits.  Host code cannot
// use the array's name as a device address; the address comes from
// cudaGetSymbolAddress, taken once per device on the first call made with
// that device current (so that first call should come before any stream
// capture).  All calls share the array and it keeps the last call's contents:
// every call first rewrites the patch table and zeroes the queue counters on
// its stream, and two calls that overlap on the GPU (different streams, or
// different host threads without ordering) race on it.  The status words in
// the array are sticky, like the library's own status word: they are read
// (OR-ed into it) by bsm_device_status and zeroed by bsm_device_status_clear.

#include <cuda_runtime.h>

#include <atomic>
#include <cstdint>
#include <mutex>

#include "bsm_internal.h"

namespace bsm {
namespace {

constexpr int64_t kNoAllocMaxPatches = BSM_NOALLOC_MAX_PATCHES;
constexpr size_t kItemsBytes = sizeof(Item) * static_cast<size_t>(kNoAllocMaxPatches);
constexpr size_t kHeadsOffset = kItemsBytes;                // 8 queue words
constexpr size_t kStatusOffset = kHeadsOffset + 8 * sizeof(uint32_t);
constexpr size_t kScratchBytes = kStatusOffset + 8 * sizeof(uint32_t);
static_assert(kItemsBytes % 256 == 0, "scratch layout");

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

struct NoAllocDevice {
    bool ready = false;
    int n_sm = 0;
    int smem_optin = 0;
    unsigned char *scratch = nullptr;   // device address of g_noalloc_scratch
};

std::mutex g_na_mu;
NoAllocDevice g_na_dev[64];

// Test-only fault injection for this entry point's launches (set through
// bsm_plan_debug with a null plan): KDEBUG_* bits and the wait bound.
std::atomic<uint32_t> g_na_debug{0};
std::atomic<uint64_t> g_na_wait_ns{0};

// Patch i covers rows [i*rpi, min((i+1)*rpi, B*R)) of the (B*R) x C matrix;
// also zero the queue counters (the status words stay: they are sticky).
__global__ void noalloc_fill(Item *items, uint32_t *heads, int64_t total_rows, int32_t R, int32_t C,
                             int32_t rpi, int32_t n_items)
{
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < 8)
        heads[i] = 0u;
    if (i >= n_items)
        return;
    const int64_t g0 = i * rpi;
    const int64_t nr = total_rows - g0 < rpi ? total_rows - g0 : rpi;
    items[i] = Item{g0 * C, C, static_cast<int32_t>(nr), static_cast<int32_t>(g0 % R), R};
}

int noalloc_device(int device, NoAllocDevice **out)
{
    if (device < 0 || device >= 64)
        return BSM_ERR_NO_DEVICE;
    std::lock_guard<std::mutex> lk(g_na_mu);
    NoAllocDevice &d = g_na_dev[device];
    if (!d.ready) {
        if (cudaDeviceGetAttribute(&d.n_sm, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
            cudaDeviceGetAttribute(&d.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, device) !=
                cudaSuccess)
            return BSM_ERR_NO_DEVICE;
        if (int e = kernel_set_smem_limit(d.smem_optin))
            return record_cuda_error(e, "cudaFuncSetAttribute");
        void *ptr = nullptr;
        if (cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch))
            return record_cuda_error(static_cast<int>(e), "cudaGetSymbolAddress");
        d.scratch = static_cast<unsigned char *>(ptr);
        d.ready = true;
    }
    *out = &d;
    return BSM_OK;
}

int softmax_noalloc(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype, uint32_t flags,
                    bsm_stream_t stream)
{
    if (B < 0 || R < 0 || C < 1 || (dtype != BSM_F32 && dtype != BSM_BF16) || (flags & ~BSM_FLAG_CAUSAL))
        return BSM_ERR_INVALID_ARG;
    if (R > INT32_MAX || C > INT32_MAX || (R > 0 && B > (int64_t(1) << 62) / R))
        return BSM_ERR_INVALID_ARG;
    const int64_t rows = B * R;
    if (rows == 0)
        return BSM_OK;
    const int es = dtype == BSM_F32 ? 4 : 2;
    const int64_t row_bytes = C * es;   // C < 2^31: no overflow
    // no two-pass path here: a row must fit one stage (checked again against
    // the device's shared memory below)
    if (row_bytes > BSM_NOALLOC_MAX_ROW_BYTES)
        return BSM_ERR_UNSUPPORTED;
    // patches of the rows that fill one stage, as the planned path cuts them
    // for large batches (device independent); the count bounds rows * C
    // before any product of them is formed
    const int64_t stage = row_bytes > kMinStageBytes ? (row_bytes + 127) & ~int64_t(127) : kMinStageBytes;
    const int64_t rpi_stage = stage / row_bytes;
    if ((rows + rpi_stage - 1) / rpi_stage > kNoAllocMaxPatches)
        return BSM_ERR_TOO_LARGE;
    if (!x || !y)
        return BSM_ERR_INVALID_ARG;
    const uintptr_t xa = reinterpret_cast<uintptr_t>(x), ya = reinterpret_cast<uintptr_t>(y);
    const uintptr_t len = static_cast<uintptr_t>(rows * row_bytes);   // < 2^16 stages of < 2^17 bytes
    if (xa != ya && xa < ya + len && ya < xa + len)
        return BSM_ERR_INVALID_ARG;
    if ((xa & 15) || (ya & 15) || row_bytes % 16 != 0)
        return BSM_ERR_MISALIGNED;
    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess)
        return BSM_ERR_NO_DEVICE;
    NoAllocDevice *nd = nullptr;
    if (int rc = noalloc_device(device, &nd))
        return rc;
    const int64_t avail = nd->smem_optin - kSmemHeader;
    if (row_bytes > ((avail / 2) & ~int64_t(127)))
        return BSM_ERR_UNSUPPORTED;
    const int n_stages = static_cast<int>(avail / stage < kMaxStages ? avail / stage : kMaxStages);
    // a small batch (fewer stage-filling patches than SMs) is cut into
    // patches of at most ceil(rows / SMs) rows, as the planned dynamic
    // schedule cuts it, so that every SM takes one
    const int64_t spread = (rows + nd->n_sm - 1) / nd->n_sm;
    const int64_t rpi = spread < rpi_stage ? (spread > 0 ? spread : 1) : rpi_stage;
    const int64_t n_items = (rows + rpi - 1) / rpi;
    if (n_items > kNoAllocMaxPatches)
        return BSM_ERR_TOO_LARGE;

    Item *items = reinterpret_cast<Item *>(nd->scratch);
    uint32_t *heads = reinterpret_cast<uint32_t *>(nd->scratch + kHeadsOffset);
    uint32_t *status = reinterpret_cast<uint32_t *>(nd->scratch + kStatusOffset);
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int threads = 256;
    const int blocks = static_cast<int>((n_items + threads - 1) / threads);
    noalloc_fill<<<blocks, threads, 0, st>>>(items, heads, rows, static_cast<int32_t>(R),
                                             static_cast<int32_t>(C), static_cast<int32_t>(rpi),
                                             static_cast<int32_t>(n_items));
    if (cudaError_t e = cudaGetLastError())
        return record_cuda_error(static_cast<int>(e), "noalloc patch fill launch");

    KernelArgs a{};
    a.x = x;
    a.y = y;
    a.total_elems = rows * C;
    a.items = items;
    a.n_items = static_cast<int32_t>(n_items);
    // at most a patch per SM: CTA u takes patch u with no claim (the static
    // deal); otherwise the device-wide queue
    a.mode = n_items <= nd->n_sm ? PULL_STATIC : PULL_QUEUE;
    a.item_begin = 0;
    a.item_end = static_cast<int32_t>(n_items);
    a.n_queues = 1;
    a.queue_begin[0] = 0;
    a.queue_len[0] = static_cast<int32_t>(n_items);
    a.steal = 0;
    a.heads = heads;
    a.sm_die = nullptr;
    a.stage_bytes = static_cast<int32_t>(stage);
    a.n_stages = n_stages;
    a.flags = flags;
    a.status = status;
    a.debug = g_na_debug.load(std::memory_order_relaxed);
    a.wait_limit_ns = g_na_wait_ns.load(std::memory_order_relaxed);
    if (int e = launch_softmax(a, dtype, OP_FORWARD, nd->n_sm, stream, false))
        return record_cuda_error(e, "noalloc kernel launch");
    return BSM_OK;
}

}  // namespace

// bsm_plan_debug(NULL, what, arg): fault injection for the launches of
// bsm_softmax_noalloc that follow (the failure-detection tests).
int noalloc_debug(int what, int64_t arg)
{
    switch (what) {
    case BSM_DEBUG_NONE:
        g_na_debug.store(0);
        g_na_wait_ns.store(0);
        return BSM_OK;
    case BSM_DEBUG_WITHHOLD_STAGE:
        if (arg <= 0)
            return BSM_ERR_INVALID_ARG;
        g_na_wait_ns.store(static_cast<uint64_t>(arg));
        g_na_debug.store(KDEBUG_WITHHOLD_STAGE0);
        return BSM_OK;
    default:
        return BSM_ERR_INVALID_ARG;
    }
}

// The sticky status bits this entry point's kernels left on `device` (0 when
// it never ran there); with clear != 0 they are zeroed afterwards.  Copies
// through the array's address, taken by the first call: nothing allocates.
// Called with the device idle (bsm_device_status synchronises it first).
int noalloc_status(int device, uint32_t *bits, int clear)
{
    *bits = 0;
    if (device < 0 || device >= 64)
        return BSM_OK;
    unsigned char *scratch = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_na_mu);
        if (g_na_dev[device].ready)
            scratch = g_na_dev[device].scratch;
    }
    if (!scratch)
        return BSM_OK;
    uint32_t *status = reinterpret_cast<uint32_t *>(scratch + kStatusOffset);
    if (cudaError_t e = cudaMemcpy(bits, status, sizeof(uint32_t), cudaMemcpyDeviceToHost))
        return record_cuda_error(static_cast<int>(e), "cudaMemcpy(noalloc status)");
    if (clear) {
        if (cudaError_t e = cudaMemset(status, 0, 8 * sizeof(uint32_t)))
            return record_cuda_error(static_cast<int>(e), "cudaMemset(noalloc status)");
    }
    return BSM_OK;
}

}  // namespace bsm

extern "C" int bsm_softmax_noalloc(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype,
                                   uint32_t flags, bsm_stream_t stream)
{
    return bsm::softmax_noalloc(x, y, B, R, C, dtype, flags, stream);
}
