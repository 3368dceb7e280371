// bsm_probe.cu -- latency probes behind the topology (Sec. 2.1: a compute
// unit reaches its nearest memory bank fastest; the latency to a farther bank
// grows with the hops in between).
//
// On GB300 each die owns half of the L2 and of the HBM stacks; an SM reading
// a line homed on the other die crosses the die-to-die link.  Both kernels
// time chains of dependent L2-only loads (ld.global.cg; each address waits
// for the previous load through an AND with a runtime zero, so it never
// depends on the data read) from one lane per SM, so the figure is the round-trip latency of an
// L2 hit from that SM to that line's home slice.
// Every loop has a fixed trip count; every address is checked against the
// buffer on the host before launch.

#include <cuda_runtime.h>
#include <cstdint>

#include "bsm_internal.h"

namespace bsm {
namespace {

__device__ __forceinline__ uint32_t probe_smid()
{
    uint32_t s;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(s));
    return s;
}

__device__ __forceinline__ uint32_t ld_l2(const uint32_t *p)
{
    uint32_t v;
    asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ long long clk()
{
    long long t;
    asm volatile("mov.u64 %0, %%clock64;" : "=l"(t));
    return t;
}

// Mean cycles of `reps` dependent L2-hit loads of the 4 bytes at p: every
// load reads p itself; its address waits for the previous load through
// "value AND zero", where zero is a kernel argument (0) the compiler cannot
// fold, so the chain never depends on the bytes read.
__device__ __forceinline__ float time_line(const unsigned char *p, int reps, uint32_t zero)
{
    const uint32_t *q = reinterpret_cast<const uint32_t *>(p);
    uint32_t v = ld_l2(q);          // brings the line into L2
    v = ld_l2(q + (v & zero));
    const long long t0 = clk();
    for (int r = 0; r < reps; ++r)
        v = ld_l2(q + (v & zero));
    const uint32_t z = v & zero;    // the clock read waits for the last load
    asm volatile("" ::"r"(z));
    const long long t1 = clk() + z;
    return static_cast<float>(t1 - t0) / reps;
}

// One CTA of 32 threads per SM does the work: the first CTA that lands on an
// SM claims it; the others return at once.
__global__ void probe_latency_kernel(const unsigned char *buf, int64_t buf_bytes, const int64_t *line_off,
                                     int n_lines, int reps, float *lat, uint32_t *claim, uint32_t zero)
{
    if (threadIdx.x != 0)
        return;
    const uint32_t sm = probe_smid() & (BSM_MAX_SM - 1);
    if (atomicCAS(&claim[sm], 0u, 1u) != 0u)
        return;
    for (int k = 0; k < n_lines; ++k) {
        const int i = static_cast<int>((k + 7ull * sm) % static_cast<unsigned>(n_lines));
        const int64_t o = line_off[i];
        if (o < 0 || o + 4 > buf_bytes || (o & 3)) {   // never true for host-checked offsets
            lat[(size_t)sm * n_lines + i] = -1.0f;
            continue;
        }
        lat[(size_t)sm * n_lines + i] = time_line(buf + o, reps, zero);
    }
}

// Latency of every `chunk`-byte chunk's first line as seen from the SMs of
// die `want_die` (the others return at once): the host compares the two
// dies' figures for each chunk, so no absolute threshold is involved.
__global__ void probe_map_kernel(const unsigned char *buf, int64_t buf_bytes, int64_t n_chunks, int64_t chunk,
                                 int reps, const int8_t *sm_die, int want_die, uint32_t *counter, float *lat_out,
                                 uint32_t zero)
{
    if (threadIdx.x != 0)
        return;
    const int my = sm_die[probe_smid() & (BSM_MAX_SM - 1)];
    if (my != want_die)
        return;
    for (int64_t guard = 0; guard < n_chunks; ++guard) {
        const uint32_t c = atomicAdd(counter, 1u);
        if (c >= n_chunks)
            break;
        if ((int64_t)c * chunk + 4 > buf_bytes)          // never true for host-checked sizes
            break;
        lat_out[c] = time_line(buf + (int64_t)c * chunk, reps, zero);
    }
}


// Die-map check: every CTA reads, from the chunks of `buf`, only those in
// the list of its own SM's die (claimed 32 at a time from that die's
// counter), each chunk once, with 16-byte L2-only loads.  With the lists
// built from an address -> die map (chunks of die d for SMs of die d), the
// L2's fabric counters then show how much of that traffic still crossed to
// the other die: none if the map is right.  The XOR of every word read goes
// to `sink` (the host checks it covers the buffer).  List entries are
// chunk indices checked on the host (< n_chunks); an index outside is
// skipped here too.
__global__ void die_check_kernel(const uint4 *buf, int64_t n_chunks, int32_t chunk_vecs,
                                 const int32_t *list0, int64_t len0, const int32_t *list1, int64_t len1,
                                 uint32_t *ctr, const int8_t *sm_die, uint32_t *sink)
{
    const int lane = threadIdx.x & 31;
    const int my = sm_die[probe_smid() & (BSM_MAX_SM - 1)];
    if (my != 0 && my != 1)
        return;
    const int32_t *list = my == 0 ? list0 : list1;
    const int64_t len = my == 0 ? len0 : len1;
    uint4 acc = make_uint4(0u, 0u, 0u, 0u);
    for (int64_t guard = 0; guard <= len / 32 + 1; ++guard) {
        uint32_t base = 0;
        if (lane == 0)
            base = atomicAdd(&ctr[my], 32u);
        base = __shfl_sync(0xFFFFFFFFu, base, 0);
        if (base >= len)
            break;
        for (int j = 0; j < 32 && base + j < len; ++j) {
            const int64_t c = list[base + j];
            if (c < 0 || c >= n_chunks)
                continue;
            const uint4 *p = buf + c * chunk_vecs;
            for (int v = lane; v < chunk_vecs; v += 32) {
                uint4 w;
                asm volatile("ld.global.cg.v4.u32 {%0, %1, %2, %3}, [%4];"
                             : "=r"(w.x), "=r"(w.y), "=r"(w.z), "=r"(w.w)
                             : "l"(p + v));
                acc.x ^= w.x;
                acc.y ^= w.y;
                acc.z ^= w.z;
                acc.w ^= w.w;
            }
        }
    }
    const uint32_t a = acc.x ^ acc.y ^ acc.z ^ acc.w;
    if (a)
        atomicXor(sink, a);
}

}  // namespace

int probe_latency_run(const void *buf, const int64_t *line_off_dev, int n_lines, int reps, int grid,
                      float *lat_dev, uint32_t *claim_dev)
{
    probe_latency_kernel<<<grid, 32>>>(static_cast<const unsigned char *>(buf), 32ll << 20, line_off_dev,
                                       n_lines, reps, lat_dev, claim_dev, 0u);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess)
        e = cudaDeviceSynchronize();
    return static_cast<int>(e);
}

int probe_map_run(const void *buf, int64_t bytes, int64_t chunk, int reps, const int8_t *sm_die_dev, int want_die,
                  int n_sm, uint32_t *counter_dev, float *lat_dev)
{
    const int64_t n_chunks = (bytes + chunk - 1) / chunk;
    // the chunk's first line must lie inside the buffer: (n_chunks-1)*chunk < bytes
    probe_map_kernel<<<n_sm, 32>>>(static_cast<const unsigned char *>(buf), bytes, n_chunks, chunk, reps,
                                   sm_die_dev, want_die, counter_dev, lat_dev, 0u);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess)
        e = cudaDeviceSynchronize();
    return static_cast<int>(e);
}

}  // namespace bsm

namespace bsm {

int die_check_run(const void *buf, int64_t n_chunks, int64_t chunk, const int32_t *list0, int64_t len0,
                  const int32_t *list1, int64_t len1, uint32_t *ctr, const int8_t *sm_die_dev, int n_sm,
                  uint32_t *sink, float *ms)
{
    cudaEvent_t e0 = nullptr, e1 = nullptr;
    cudaEventCreate(&e0);
    cudaEventCreate(&e1);
    cudaEventRecord(e0);
    die_check_kernel<<<n_sm, 256>>>(static_cast<const uint4 *>(buf), n_chunks, static_cast<int32_t>(chunk / 16),
                                    list0, len0, list1, len1, ctr, sm_die_dev, sink);
    cudaError_t e = cudaGetLastError();
    cudaEventRecord(e1);
    if (e == cudaSuccess)
        e = cudaDeviceSynchronize();
    if (e == cudaSuccess && ms)
        cudaEventElapsedTime(ms, e0, e1);
    cudaEventDestroy(e0);
    cudaEventDestroy(e1);
    return static_cast<int>(e);
}

}  // namespace bsm
