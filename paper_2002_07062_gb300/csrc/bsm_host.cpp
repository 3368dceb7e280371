// bsm_host.cpp -- bsm_softmax_host: the batched softmax on HOST buffers.
//
// Page-locked (pinned) buffers are read and written by the kernel itself:
// on Grace-Blackwell the GPU reaches host memory over NVLink-C2C, so the
// bulk copies of the patches come straight from x_host and the stores go
// straight to y_host -- no staging memory, both link directions busy at once.
//
// Pageable buffers go through a staged pipeline: the batch is cut into
// chunks of whole slices; every chunk goes through three stages on three
// streams of the library -- copy in (host to device), the softmax kernel (the
// plan-cached bsm_softmax_ex path on a device staging buffer), copy out
// (device to host) -- with two staging buffers.  A device-to-host copy into
// pageable memory returns to the host only once it has finished, so the
// host thread issues chunk i's copy-in and kernel before chunk i-1's
// copy-out: while the host waits on that copy-out, chunk i moves in and is
// computed.  Both link directions are then busy at once, but only in pairs
// of chunks (the copy-in of chunk i+1 is issued after chunk i-1's copy-out
// has finished), and the driver stages pageable copies through its own
// buffers; pinned buffers are the fast path.

#include <cuda_runtime.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "bsm_internal.h"
#include "bsm_trace.h"

namespace bsm {
namespace {

constexpr int64_t kChunkBytes = 48ll << 20;   // input bytes per chunk (target)

struct HostPipe {
    bool ready = false;
    cudaStream_t s_in = nullptr, s_k = nullptr, s_out = nullptr;
    cudaEvent_t ev_start = nullptr, ev_end = nullptr;
    cudaEvent_t ev_in[2] = {nullptr, nullptr}, ev_k[2] = {nullptr, nullptr},
                ev_out[2] = {nullptr, nullptr};
    bool out_recorded[2] = {false, false};
    void *dx[2] = {nullptr, nullptr}, *dy[2] = {nullptr, nullptr};
    int64_t cap = 0;   // bytes of each staging buffer
};

std::mutex g_host_mu;
HostPipe g_pipe[64];

int pipe_init(HostPipe &p)
{
    if (p.ready)
        return BSM_OK;
    cudaError_t e = cudaSuccess;
    auto ok = [&](cudaError_t r) { e = r; return r == cudaSuccess; };
    if (!ok(cudaStreamCreateWithFlags(&p.s_in, cudaStreamNonBlocking)) ||
        !ok(cudaStreamCreateWithFlags(&p.s_k, cudaStreamNonBlocking)) ||
        !ok(cudaStreamCreateWithFlags(&p.s_out, cudaStreamNonBlocking)) ||
        !ok(cudaEventCreateWithFlags(&p.ev_start, cudaEventDisableTiming)) ||
        !ok(cudaEventCreateWithFlags(&p.ev_end, cudaEventDisableTiming)))
        return record_cuda_error(static_cast<int>(e), "host pipeline streams");
    for (int b = 0; b < 2; ++b)
        if (!ok(cudaEventCreateWithFlags(&p.ev_in[b], cudaEventDisableTiming)) ||
            !ok(cudaEventCreateWithFlags(&p.ev_k[b], cudaEventDisableTiming)) ||
            !ok(cudaEventCreateWithFlags(&p.ev_out[b], cudaEventDisableTiming)))
            return record_cuda_error(static_cast<int>(e), "host pipeline events");
    p.ready = true;
    return BSM_OK;
}

int pipe_reserve(HostPipe &p, int64_t bytes)
{
    if (bytes <= p.cap)
        return BSM_OK;
    // buffers may still be in use by an earlier call
    if (cudaError_t e = cudaStreamSynchronize(p.s_out))
        return record_cuda_error(static_cast<int>(e), "host pipeline sync");
    for (int b = 0; b < 2; ++b) {
        cudaFree(p.dx[b]);
        cudaFree(p.dy[b]);
        p.dx[b] = p.dy[b] = nullptr;
    }
    p.cap = 0;
    for (int b = 0; b < 2; ++b) {
        if (cudaMalloc(&p.dx[b], static_cast<size_t>(bytes)) != cudaSuccess ||
            cudaMalloc(&p.dy[b], static_cast<size_t>(bytes)) != cudaSuccess)
            return BSM_ERR_NOMEM;
    }
    p.cap = bytes;
    return BSM_OK;
}

int softmax_host(const void *x_host, void *y_host, int64_t B, int64_t R, int64_t C, int dtype, int policy,
                 uint32_t flags, bsm_stream_t stream)
{
    TraceRange trace("bsm_softmax_host");
    if (B < 0 || R < 0 || C < 1 || (dtype != BSM_F32 && dtype != BSM_BF16) || (flags & ~BSM_FLAG_CAUSAL) ||
        policy < BSM_POLICY_WHOLE_GPU || policy > BSM_POLICY_MINIMAX)
        return BSM_ERR_INVALID_ARG;
    if (R > INT32_MAX || C > INT32_MAX || (R > 0 && B > (int64_t(1) << 40) / R))
        return BSM_ERR_INVALID_ARG;
    if (B == 0 || R == 0)
        return BSM_OK;
    if (!x_host || !y_host)
        return BSM_ERR_INVALID_ARG;
    const int es = dtype == BSM_F32 ? 4 : 2;
    if ((C * es) % 16)
        return BSM_ERR_MISALIGNED;
    const int64_t slice_bytes = R * C * es;
    if (slice_bytes > (int64_t(1) << 40) / std::max<int64_t>(1, B))
        return BSM_ERR_INVALID_ARG;
    const uintptr_t xa = reinterpret_cast<uintptr_t>(x_host), ya = reinterpret_cast<uintptr_t>(y_host);
    const uintptr_t len = static_cast<uintptr_t>(B * slice_bytes);
    if (xa != ya && xa < ya + len && ya < xa + len)
        return BSM_ERR_INVALID_ARG;
    // pinned host memory: the kernel accesses it directly
    cudaPointerAttributes ax{}, ay{};
    if (cudaPointerGetAttributes(&ax, x_host) == cudaSuccess &&
        cudaPointerGetAttributes(&ay, y_host) == cudaSuccess && ax.type == cudaMemoryTypeHost &&
        ay.type == cudaMemoryTypeHost && ax.devicePointer && ay.devicePointer)
        return bsm_softmax_ex(ax.devicePointer, ay.devicePointer, B, R, C, dtype, policy, flags, stream);
    cudaGetLastError();   // a pageable pointer is not an error here

    const int64_t per_chunk = std::max<int64_t>(1, std::min<int64_t>(B, kChunkBytes / slice_bytes));
    const int64_t chunk_bytes = per_chunk * slice_bytes;

    int device = 0;
    if (cudaGetDevice(&device) != cudaSuccess || device < 0 || device >= 64)
        return BSM_ERR_NO_DEVICE;
    std::lock_guard<std::mutex> lk(g_host_mu);
    HostPipe &p = g_pipe[device];
    if (int rc = pipe_init(p))
        return rc;
    if (int rc = pipe_reserve(p, (chunk_bytes + 255) & ~int64_t(255)))
        return rc;
    cudaStream_t caller = reinterpret_cast<cudaStream_t>(stream);
    cudaError_t e;
    if ((e = cudaEventRecord(p.ev_start, caller)) || (e = cudaStreamWaitEvent(p.s_in, p.ev_start, 0)) ||
        (e = cudaStreamWaitEvent(p.s_k, p.ev_start, 0)) || (e = cudaStreamWaitEvent(p.s_out, p.ev_start, 0)))
        return record_cuda_error(static_cast<int>(e), "host pipeline start");
    const unsigned char *xs = static_cast<const unsigned char *>(x_host);
    unsigned char *ys = static_cast<unsigned char *>(y_host);
    // copy-out of a computed chunk (staging buffer b, its place in y); it
    // waits for that chunk's kernel only (ev_k[b], recorded after it)
    auto copy_out = [&](int b, int64_t off, int64_t bytes) -> int {
        cudaError_t ee;
        if ((ee = cudaStreamWaitEvent(p.s_out, p.ev_k[b], 0)) ||
            (ee = cudaMemcpyAsync(ys + off, p.dy[b], static_cast<size_t>(bytes), cudaMemcpyDeviceToHost,
                                  p.s_out)) ||
            (ee = cudaEventRecord(p.ev_out[b], p.s_out)))
            return record_cuda_error(static_cast<int>(ee), "host pipeline copy out");
        p.out_recorded[b] = true;
        return BSM_OK;
    };
    int pend_b = -1;                 // the chunk computed but not yet copied out
    int64_t pend_off = 0, pend_bytes = 0;
    for (int64_t first = 0, i = 0; first < B; first += per_chunk, ++i) {
        const int b = static_cast<int>(i & 1);
        const int64_t n = std::min<int64_t>(per_chunk, B - first);
        const int64_t bytes = n * slice_bytes;
        const int64_t off = first * slice_bytes;
        // the staging buffer is free once its previous copy-out finished
        if (p.out_recorded[b] && (e = cudaStreamWaitEvent(p.s_in, p.ev_out[b], 0)))
            return record_cuda_error(static_cast<int>(e), "host pipeline wait");
        if ((e = cudaMemcpyAsync(p.dx[b], xs + off, static_cast<size_t>(bytes), cudaMemcpyHostToDevice,
                                 p.s_in)) ||
            (e = cudaEventRecord(p.ev_in[b], p.s_in)) || (e = cudaStreamWaitEvent(p.s_k, p.ev_in[b], 0)))
            return record_cuda_error(static_cast<int>(e), "host pipeline copy in");
        if (int rc = bsm_softmax_ex(p.dx[b], p.dy[b], n, R, C, dtype, policy, flags,
                                    reinterpret_cast<bsm_stream_t>(p.s_k)))
            return rc;
        if ((e = cudaEventRecord(p.ev_k[b], p.s_k)))
            return record_cuda_error(static_cast<int>(e), "host pipeline kernel");
        // the previous chunk's copy-out after this chunk's copy-in and kernel
        // are queued (it may block the host until it has finished)
        if (pend_b >= 0)
            if (int rc = copy_out(pend_b, pend_off, pend_bytes))
                return rc;
        pend_b = b;
        pend_off = off;
        pend_bytes = bytes;
    }
    if (pend_b >= 0)
        if (int rc = copy_out(pend_b, pend_off, pend_bytes))
            return rc;
    if ((e = cudaEventRecord(p.ev_end, p.s_out)) || (e = cudaStreamWaitEvent(caller, p.ev_end, 0)))
        return record_cuda_error(static_cast<int>(e), "host pipeline end");
    return BSM_OK;
}

}  // namespace
}  // namespace bsm

extern "C" int bsm_softmax_host(const void *x_host, void *y_host, int64_t B, int64_t R, int64_t C, int dtype,
                                int policy, uint32_t flags, bsm_stream_t stream)
{
    try {
        return bsm::softmax_host(x_host, y_host, B, R, C, dtype, policy, flags, stream);
    } catch (...) {
        return BSM_ERR_NOMEM;
    }
}
