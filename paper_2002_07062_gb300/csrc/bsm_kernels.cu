// bsm_kernels.cu -- the persistent batched-softmax kernel for sm_103a.
//
// One CTA per SM.  Warp 16 is the producer: one lane pulls the next patch
// (Sec. 4: a block of rows of one slice) from the schedule -- a static list
// for the Sec. 3 baselines, or the CTA's die queue for Cluster Beamforming
// (Sec. 4.1) with stealing after the Sec. 4.2 balance -- and streams the
// patch's contiguous bytes into a ring of shared-memory stages with one 1-D
// TMA bulk copy (cp.async.bulk, completion counted on an mbarrier).  Warps
// 0..15 are consumers: they wait on a stage's "full" barrier, compute the
// softmax of its rows out of shared memory, store y with 128-bit coalesced
// stores, and release the stage on its "empty" barrier.  The patch geometry
// travels with the stage (the "templated kernel fed patch coordinates from a
// queue" of Sec. 5).
//
// Row routine (the arithmetic, identical under every policy): a row is owned
// by a group of T lanes; lane l owns the 16-byte vectors l, l + T, l + 2T, ...
// The maximum and the sum are per vector (a balanced tree), per lane in vector
// order, then a butterfly (xor) shuffle tree over the group.  By row length in
// 16-byte vectors: <= 8: T = 8, 1 vector per lane; <= 16: T = 8, 2; <= 32:
// T = 8, 4; <= 64: T = 16, 4; <= 128: T = 32, 4; fp32 <= 256: T = 32, 8 -- all
// in registers (at most 32 elements per lane); longer fp32 rows: one warp,
// exponentials written back in place in shared memory; longer bf16 rows: one
// warp, three sweeps over shared memory (max, sum, write).  exp(t) is evaluated as 2^(t*log2 e) with
// the exponent formed by one fused multiply-add, v*log2e - m*log2e, and the
// power of two from the PTX ex2.approx instruction; y = p * (1/sum).
//
// Every wait is bounded (2 s of wall time unless the launch asks for less):
// on expiry the CTA
// records BSM_DEV_TIMEOUT in the status word, lets its copies in flight land,
// and returns.

#include <cuda_runtime.h>
#include <cstdint>

#include "bsm_internal.h"

namespace bsm {
namespace {

constexpr uint64_t kWaitLimitNs = 2000000000ull;   // 2 s
constexpr uint32_t kClaimAhead = 2;                 // rows a group's rank 0 announces ahead
constexpr float kLog2e = 1.4426950408889634f;

enum : int32_t { KIND_DATA = 0, KIND_SKIP = 1, KIND_DONE = 2, KIND_LONG = 3, KIND_GROUP = 4 };

struct alignas(16) StageMeta {
    int64_t off;
    int32_t C;          // KIND_LONG: elements of this chunk of the row
    int32_t nrows;
    int32_t row0;
    int32_t kind;
    int32_t R;
    int32_t col0;       // KIND_LONG: column of the chunk's first element
    int32_t pass;       // KIND_LONG: 0 = partial of the segment, 1 = combine and write
    int32_t last;       // KIND_LONG: last chunk of the segment
    int32_t first;      // KIND_LONG: first chunk of the segment
    int32_t part;       // KIND_LONG: the segment's partial slot
    int32_t part_first; // KIND_LONG: the row's first partial slot
    int32_t part_count; // KIND_LONG: the row's number of segments
    int32_t resident;   // KIND_LONG: the whole row stays staged for its second pass
    int32_t pad;
};
static_assert(sizeof(StageMeta) == 64, "StageMeta layout");

struct SmemHeader {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t xwarp;                 // long rows: the consumer warps' partials are in
    uint32_t xarrive[2];            // rows over groups: warps whose partial is in, by row parity
    StageMeta meta[kMaxStages];
    float2 partial[2][kConsumerWarps];   // long rows: (max, sum) per warp, two rows deep
    int32_t abort_flag;
};
static_assert(sizeof(SmemHeader) <= kSmemHeader, "header too large");

// ---------------------------------------------------------------- PTX helpers

__device__ __forceinline__ uint32_t smem_addr(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t global_timer_ns()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ uint32_t sm_id()
{
    uint32_t s;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(s));
    return s;
}

__device__ __forceinline__ void mbar_init(uint64_t *bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(bar)), "r"(count)
                 : "memory");
}

__device__ __forceinline__ void mbar_init_fence()
{
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t *bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_addr(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t *bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(bar)),
                 "r"(bytes)
                 : "memory");
}

// One potentially blocking test of the phase: a waiting thread is suspended
// in hardware (it issues nothing) until the phase completes or kSuspendNs
// pass, so idle warps do not take issue slots from the working ones.
constexpr uint32_t kSuspendNs = 50000;

__device__ __forceinline__ bool mbar_try_wait(uint64_t *bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(smem_addr(bar)), "r"(parity), "r"(kSuspendNs)
        : "memory");
    return ok != 0;
}

// Wait until the phase with the given parity of `bar` has completed.  Gives
// up (returns false) when *abort becomes non-zero (if abort != nullptr) or
// after limit_ns.
__device__ __noinline__ bool mbar_wait_bounded(uint64_t *bar, uint32_t parity,
                                               const volatile int32_t *abort, uint64_t limit_ns)
{
    if (mbar_try_wait(bar, parity))
        return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < (1u << 28); ++it) {
        if (mbar_try_wait(bar, parity))
            return true;
        {
            if (abort && *abort)
                return false;
            if (global_timer_ns() - t0 > limit_ns)
                return false;
        }
    }
    return false;
}

// 1-D bulk copy global -> shared, completion counted (bytes) on `bar`.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t bytes, uint64_t *bar)
{
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
            smem_addr(dst)),
        "l"(src), "r"(bytes), "r"(smem_addr(bar))
        : "memory");
}

// Stage reads and in-place writes are explicit shared-space accesses (a
// 32-bit shared address), so they are issued as shared loads/stores whatever
// the compiler can infer about the pointer; volatile keeps them on their side
// of the barrier waits.
__device__ __forceinline__ uint4 lds128(const unsigned char *p)
{
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(smem_addr(p)));
    return v;
}

__device__ __forceinline__ void sts128(unsigned char *p, uint4 v)
{
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(smem_addr(p)), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
}

// Output stores: plain 128-bit global stores.
__device__ __forceinline__ void stg128(void *p, uint4 v)
{
    *reinterpret_cast<uint4 *>(p) = v;
}

// ---------------------------------------------------------- self-checks
// The checking instantiation (Checked = true) verifies every shared-memory
// read, global store and bulk copy against the stage and buffer extents; a
// violation is recorded (BSM_DEV_CHECK, plus the first one's details in words
// 1..7 of the status block) and the access is skipped.

struct Bounds {
    const unsigned char *s_lo, *s_hi;   // bytes of the current stage that hold the patch
    const unsigned char *y_lo, *y_hi;   // the output buffer
    uint32_t *status;
};

__device__ __noinline__ void check_fail(uint32_t *status, uint32_t kind, uint64_t a, uint64_t b)
{
    atomicOr(status, BSM_DEV_CHECK);
    if (atomicCAS(&status[1], 0u, kind) == 0u) {
        status[2] = blockIdx.x;
        status[3] = threadIdx.x;
        status[4] = static_cast<uint32_t>(a);
        status[5] = static_cast<uint32_t>(a >> 32);
        status[6] = static_cast<uint32_t>(b);
        status[7] = static_cast<uint32_t>(b >> 32);
    }
}

template <bool Checked>
__device__ __forceinline__ bool load_vec(const unsigned char *p, const Bounds &b, uint4 &out)
{
    if (Checked && (p < b.s_lo || p + 16 > b.s_hi || (reinterpret_cast<uintptr_t>(p) & 15))) {
        check_fail(b.status, 1, static_cast<uint64_t>(p - b.s_lo), static_cast<uint64_t>(b.s_hi - b.s_lo));
        return false;
    }
    out = lds128(p);
    return true;
}

template <bool Checked>
__device__ __forceinline__ void store_vec(unsigned char *p, const Bounds &b, uint4 v)
{
    if (Checked && (p < b.y_lo || p + 16 > b.y_hi || (reinterpret_cast<uintptr_t>(p) & 15))) {
        check_fail(b.status, 2, static_cast<uint64_t>(p - b.y_lo), static_cast<uint64_t>(b.y_hi - b.y_lo));
        return;
    }
    stg128(p, v);
}

__device__ __forceinline__ float ex2(float a)
{
    float r;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(a));
    return r;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// ------------------------------------------------------- element-type traits

template <typename Tag> struct Elem;
struct F32 {};
struct BF16 {};

template <> struct Elem<F32> {
    static constexpr int kSize = 4;
    static constexpr int kPerVec = 4;
    __device__ static __forceinline__ void unpack(uint4 r, float (&v)[4])
    {
        v[0] = __uint_as_float(r.x);
        v[1] = __uint_as_float(r.y);
        v[2] = __uint_as_float(r.z);
        v[3] = __uint_as_float(r.w);
    }
    __device__ static __forceinline__ uint4 pack(const float (&v)[4])
    {
        return make_uint4(__float_as_uint(v[0]), __float_as_uint(v[1]), __float_as_uint(v[2]),
                          __float_as_uint(v[3]));
    }
    // a vector of -inf (stands in for vectors past the end of a row)
    __device__ static __forceinline__ uint4 neg_inf_vec() { return make_uint4(0xFF800000u, 0xFF800000u, 0xFF800000u, 0xFF800000u); }
};

template <> struct Elem<BF16> {
    static constexpr int kSize = 2;
    static constexpr int kPerVec = 8;
    __device__ static __forceinline__ void unpack(uint4 r, float (&v)[8])
    {
        const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            v[2 * k] = __uint_as_float(w[k] << 16);
            v[2 * k + 1] = __uint_as_float(w[k] & 0xFFFF0000u);
        }
    }
    __device__ static __forceinline__ uint4 pack(const float (&v)[8])
    {
        return make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]),
                          pack_bf16x2(v[6], v[7]));
    }
    __device__ static __forceinline__ uint4 neg_inf_vec() { return make_uint4(0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u, 0xFF80FF80u); }
};

// ------------------------------------------------------------- row routines

template <int T> __device__ __forceinline__ float group_max(float m)
{
#pragma unroll
    for (int o = T / 2; o >= 1; o >>= 1)
        m = fmaxf(m, __shfl_xor_sync(0xFFFFFFFFu, m, o));
    return m;
}

template <int T> __device__ __forceinline__ float group_sum(float s)
{
#pragma unroll
    for (int o = T / 2; o >= 1; o >>= 1)
        s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    return s;
}

// Maximum / sum of the N elements of one vector as a balanced tree (fixed
// order: the sum's rounding is the same wherever the row runs).
template <int N> __device__ __forceinline__ float tree_max(const float *v)
{
    if constexpr (N == 1)
        return v[0];
    else
        return fmaxf(tree_max<N / 2>(v), tree_max<N / 2>(v + N / 2));
}

template <int N> __device__ __forceinline__ float tree_sum(const float *v)
{
    if constexpr (N == 1)
        return v[0];
    else
        return tree_sum<N / 2>(v) + tree_sum<N / 2>(v + N / 2);
}

// p = exp(v - m) for one vector, as 2^(v*log2e - m*log2e).  For a vector
// lying wholly above the causal diagonal (v is x, or x + (-inf)) the formula
// gives 0 where x is finite or -inf and NaN where x is NaN or +inf; that is
// computed without the exponential.
template <int EPV>
__device__ __forceinline__ void vec_exp(float (&v)[EPV], float mL, bool masked)
{
    if (masked) {
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            v[e] = v[e] < INFINITY ? 0.0f : __int_as_float(0x7FC00000);
    } else {
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            v[e] = ex2(fmaf(v[e], kLog2e, -mL));
    }
}

// Additive causal mask of one 16-byte vector: element c of the row gets -inf
// when c > row.
template <int EPV>
__device__ __forceinline__ void apply_causal(float (&v)[EPV], int col0, int row)
{
#pragma unroll
    for (int e = 0; e < EPV; ++e)
        v[e] += (col0 + e > row) ? -INFINITY : 0.0f;
}

// Register-resident fp32 row: T lanes, up to V vectors per lane, scalar
// arithmetic (fp32 rows move 8 bytes per element: memory, not instruction
// issue, bounds them).  Under the causal mask a vector is unmasked (all its
// columns <= row), on the diagonal (masked element by element) or wholly
// masked (it adds nothing to the max; its p is 0 or NaN, see vec_exp).
template <typename Tag, bool Checked, int T, int V>
__device__ __forceinline__ void row_in_registers_scalar(const unsigned char *srow, unsigned char *yrow,
                                                 int nvec, int row, bool causal, int l, bool valid,
                                                 const Bounds &bd)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    float v[V][EPV];
    float m = -INFINITY;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        const bool masked = causal && vi * EPV > row;
        uint4 raw;
        if (valid && vi < nvec && load_vec<Checked>(srow + 16 * vi, bd, raw)) {
            E::unpack(raw, v[j]);
            if (!masked) {
                if (causal && vi * EPV + EPV - 1 > row)
                    apply_causal<EPV>(v[j], vi * EPV, row);
                m = fmaxf(m, tree_max<EPV>(v[j]));
            }
        } else {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                v[j][e] = -INFINITY;
        }
    }
    m = group_max<T>(m);
    const float mL = m * kLog2e;
    float s = 0.0f;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        vec_exp<EPV>(v[j], mL, (causal && vi * EPV > row) || vi >= nvec);
        if (vi < nvec)
            s += tree_sum<EPV>(v[j]);
    }
    s = group_sum<T>(s);
    const float inv = __frcp_rn(s);
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        if (valid && vi < nvec) {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                v[j][e] *= inv;
            store_vec<Checked>(yrow + 16 * vi, bd, E::pack(v[j]));
        }
    }
}

// ------------------------------------------------ fp32 pair arithmetic
// One instruction, two IEEE operations, each rounded like its scalar form.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c)
{
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}

__device__ __forceinline__ float2 add2(float2 a, float2 b)
{
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

__device__ __forceinline__ float2 mul2(float2 a, float2 b)
{
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

// p = 2^(v*log2e - mL) for one vector, in pairs; returns the vector's sum as
// a pair: ((p0,p1) + (p2,p3)) [+ ((p4,p5) + (p6,p7))].
template <int EPV>
__device__ __forceinline__ float2 vec_exp_pairs(float (&v)[EPV], float mL)
{
    const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-mL, -mL);
#pragma unroll
    for (int e = 0; e < EPV; e += 2) {
        const float2 t = fma2(make_float2(v[e], v[e + 1]), l2, nm);
        v[e] = ex2(t.x);
        v[e + 1] = ex2(t.y);
    }
    const float2 a = add2(make_float2(v[0], v[1]), make_float2(v[2], v[3]));
    if constexpr (EPV == 4)
        return a;
    else
        return add2(a, add2(make_float2(v[4], v[5]), make_float2(v[6], v[7])));
}

// Element-wise maximum of two bf16 pairs.
__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b)
{
    uint32_t d;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
    return d;
}

// True when one of the vector's elements is NaN or +inf (such an element
// masked by the causal mask still turns its row into NaN: NaN + (-inf) and
// +inf + (-inf) are NaN); a NaN-propagating maximum over the raw vector.
template <typename Tag> __device__ __forceinline__ bool vec_poisons(uint4 r);
template <> __device__ __forceinline__ bool vec_poisons<BF16>(uint4 r)
{
    uint32_t w;
    asm("{\n\t.reg .b32 a, b;\n\tmax.NaN.bf16x2 a, %1, %2;\n\tmax.NaN.bf16x2 b, %3, %4;\n\t"
        "max.NaN.bf16x2 %0, a, b;\n\t}"
        : "=r"(w)
        : "r"(r.x), "r"(r.y), "r"(r.z), "r"(r.w));
    const float lo = __uint_as_float(w << 16), hi = __uint_as_float(w & 0xFFFF0000u);
    return !(lo < INFINITY) || !(hi < INFINITY);
}

// p = 2^(v*log2e - mL) for one vector in fp32 pairs (each pair two IEEE
// fmas: the bits of vec_exp), and the vector's sum in tree_sum's order
// ((p0 + p1) + (p2 + p3), and so on).
template <int EPV>
__device__ __forceinline__ float vec_exp_sum_pairs(float (&v)[EPV], float mL)
{
    const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-mL, -mL);
#pragma unroll
    for (int e = 0; e < EPV; e += 2) {
        const float2 t = fma2(make_float2(v[e], v[e + 1]), l2, nm);
        v[e] = ex2(t.x);
        v[e + 1] = ex2(t.y);
    }
    if constexpr (EPV == 4) {
        const float2 a = add2(make_float2(v[0], v[2]), make_float2(v[1], v[3]));
        return a.x + a.y;
    } else {
        const float2 a = add2(make_float2(v[0], v[4]), make_float2(v[1], v[5]));
        const float2 b = add2(make_float2(v[2], v[6]), make_float2(v[3], v[7]));
        const float2 c = add2(a, b);
        return c.x + c.y;
    }
}

// The maximum of a chunk's vectors as loaded: bf16 on the packed words
// (exact; a NaN operand loses, as with fmaxf), fp32 through tree_max.
template <typename Tag, int N>
__device__ __forceinline__ float raw_max(const uint4 (&raw)[N], const float (&v)[N][Elem<Tag>::kPerVec])
{
    if constexpr (Elem<Tag>::kSize == 2) {
        uint32_t mw = 0xFF80FF80u;
#pragma unroll
        for (int j = 0; j < N; ++j)
            mw = bmax2(mw, bmax2(bmax2(raw[j].x, raw[j].y), bmax2(raw[j].z, raw[j].w)));
        return fmaxf(__uint_as_float(mw << 16), __uint_as_float(mw & 0xFFFF0000u));
    } else {
        float m = -INFINITY;
#pragma unroll
        for (int j = 0; j < N; ++j)
            m = fmaxf(m, tree_max<Elem<Tag>::kPerVec>(v[j]));
        return m;
    }
}

// Register-resident bf16 row (bf16 rows move 4 bytes per element, so
// instruction issue matters): T lanes, V vectors per lane (vector j of lane l
// is vector j*T + l of the row).  Arithmetic, the same in both variants and
// under every policy: m = max over the lane's vectors (balanced tree per
// vector, vectors in order), butterfly over the lane group; p = 2^(v*log2e
// - m*log2e) in fp32 pairs; the lane's sum is a pair accumulated vector by
// vector, then its two halves, then the butterfly; y = p * (1/sum).
// Full = true: every lane holds V vectors of a valid row and nothing needs a
// bound (no per-vector predicates).  Under the causal mask each vector is
// classed for the whole warp: unmasked everywhere (no mask work), masked
// everywhere (p = 0 without an exponential; a NaN or +inf among its inputs
// still makes the row NaN), or mixed (the additive -inf mask element by
// element).  Results do not depend on the class: the mask's sums are exact.
template <typename Tag, bool Checked, int T, int V, bool Full>
__device__ __forceinline__ void row_in_registers_pairs(const unsigned char *srow, unsigned char *yrow,
                                                 int nvec, int row, bool causal, int l, bool valid,
                                                 const Bounds &bd)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    float v[V][EPV];
    uint32_t skip = 0;          // bit j: vector j is masked for the whole warp
    bool poison = false;
    float m = -INFINITY;
    uint32_t mw = 0xFF80FF80u;  // running maximum of the unmasked vectors, two bf16 halves
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        const int col0 = vi * EPV;
        const bool in = Full || (valid && vi < nvec);
        // the vector's mask class depends on its position only (warp-wide)
        bool mixed = false;
        if (causal) {
            const bool lane_un = !in || col0 + EPV - 1 <= row;
            const bool lane_mk = !in || col0 > row;
            if (!__all_sync(0xFFFFFFFFu, lane_un)) {
                if (__all_sync(0xFFFFFFFFu, lane_mk))
                    skip |= 1u << j;
                else
                    mixed = true;
            }
        }
        uint4 raw = E::neg_inf_vec();
        if (Full) {
            raw = lds128(srow + 16 * vi);
        } else if (in) {
            uint4 r;
            if (load_vec<Checked>(srow + 16 * vi, bd, r))
                raw = r;
        }
        if (skip & (1u << j)) {
            if (in)
                poison |= vec_poisons<Tag>(raw);
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                v[j][e] = 0.0f;
            continue;
        }
        E::unpack(raw, v[j]);
        if (mixed) {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                v[j][e] += (col0 + e > row) ? -INFINITY : 0.0f;
            m = fmaxf(m, tree_max<EPV>(v[j]));
        } else {
            // the maximum of bf16 values is exact in bf16: take it on the
            // packed words (non-NaN operand wins, as fmaxf), unpack once
            mw = bmax2(mw, bmax2(bmax2(raw.x, raw.y), bmax2(raw.z, raw.w)));
        }
    }
    m = fmaxf(m, fmaxf(__uint_as_float(mw << 16), __uint_as_float(mw & 0xFFFF0000u)));
    m = group_max<T>(m);
    const float mL = m * kLog2e;
    float2 acc = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int j = 0; j < V; ++j)
        if (!(skip & (1u << j)))
            acc = add2(acc, vec_exp_pairs<EPV>(v[j], mL));
    float s = acc.x + acc.y;
    if (poison)
        s = __int_as_float(0x7FC00000);
    s = group_sum<T>(s);
    const float inv = __frcp_rn(s);
    const float2 inv2 = make_float2(inv, inv);
    const float zero_y = 0.0f * inv;   // the output of a masked element (0, or NaN in a NaN row)
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        if (Full || (valid && vi < nvec)) {
            if (skip & (1u << j)) {
#pragma unroll
                for (int e = 0; e < EPV; ++e)
                    v[j][e] = zero_y;
            } else {
#pragma unroll
                for (int e = 0; e < EPV; e += 2) {
                    const float2 y2 = mul2(make_float2(v[j][e], v[j][e + 1]), inv2);
                    v[j][e] = y2.x;
                    v[j][e + 1] = y2.y;
                }
            }
            store_vec<Checked>(yrow + 16 * vi, bd, E::pack(v[j]));
        }
    }
}

// Shared-memory-resident row of any length: one warp, three sweeps (max;
// exponentials and their sum; exponentials again, scaled, stored).
template <typename Tag, bool Checked>
__device__ __forceinline__ void row_in_smem(const unsigned char *srow, unsigned char *yrow, int nvec,
                                            int row, bool causal, int lane, const Bounds &bd)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    float v[EPV];
    uint4 raw;
    float m = -INFINITY;
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
        if (causal)
            apply_causal<EPV>(v, vi * EPV, row);
        m = fmaxf(m, tree_max<EPV>(v));
    }
    m = group_max<32>(m);
    const float mL = m * kLog2e;
    float s = 0.0f;
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
        if (causal)
            apply_causal<EPV>(v, vi * EPV, row);
        vec_exp<EPV>(v, mL, causal && vi * EPV > row);
        s += tree_sum<EPV>(v);
    }
    s = group_sum<32>(s);
    const float inv = __frcp_rn(s);
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
        if (causal)
            apply_causal<EPV>(v, vi * EPV, row);
        vec_exp<EPV>(v, mL, causal && vi * EPV > row);
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            v[e] *= inv;
        store_vec<Checked>(yrow + 16 * vi, bd, E::pack(v));
    }
}

// fp32 rows of any length, two exponential-free sweeps: the second sweep
// writes p = exp(v - m) back over the row in shared memory (same size as x),
// the third scales it.  One exponential per element.  The proxy fence orders
// these generic writes before the bulk copy that later refills the stage.
template <bool Checked>
__device__ __forceinline__ void row_in_smem_inplace(unsigned char *srow, unsigned char *yrow, int nvec,
                                                    int row, bool causal, int lane, const Bounds &bd)
{
    using E = Elem<F32>;
    constexpr int EPV = E::kPerVec;
    float v[EPV];
    uint4 raw;
    float m = -INFINITY;
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
        if (causal)
            apply_causal<EPV>(v, vi * EPV, row);
        m = fmaxf(m, tree_max<EPV>(v));
    }
    m = group_max<32>(m);
    const float mL = m * kLog2e;
    float s = 0.0f;
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
        if (causal)
            apply_causal<EPV>(v, vi * EPV, row);
        vec_exp<EPV>(v, mL, causal && vi * EPV > row);
        s += tree_sum<EPV>(v);
        sts128(srow + 16 * vi, E::pack(v));
    }
    s = group_sum<32>(s);
    const float inv = __frcp_rn(s);
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(srow + 16 * vi, bd, raw))
            continue;
        E::unpack(raw, v);
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            v[e] *= inv;
        store_vec<Checked>(yrow + 16 * vi, bd, E::pack(v));
    }
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------------ backward row routines
// dx = y * (dy - <y, dy>) of one row; y and dy sit in the two halves of the
// stage.  The dot product: per vector a balanced tree of y*dy, per lane in
// vector order, then the butterfly over the lane group.

template <typename Tag, bool Checked, int T, int V>
__device__ __forceinline__ void row_bwd_registers(const unsigned char *sy, const unsigned char *sdy,
                                                  unsigned char *dxrow, int nvec, int l, bool valid,
                                                  const Bounds &by, const Bounds &bdy)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    float yv[V][EPV], dv[V][EPV];
    float dot = 0.0f;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        uint4 ry, rd;
        if (valid && vi < nvec && load_vec<Checked>(sy + 16 * vi, by, ry) &&
            load_vec<Checked>(sdy + 16 * vi, bdy, rd)) {
            E::unpack(ry, yv[j]);
            E::unpack(rd, dv[j]);
            float pr[EPV];
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                pr[e] = yv[j][e] * dv[j][e];
            dot += tree_sum<EPV>(pr);
        } else {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                yv[j][e] = dv[j][e] = 0.0f;
        }
    }
    dot = group_sum<T>(dot);
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const int vi = j * T + l;
        if (valid && vi < nvec) {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                yv[j][e] = yv[j][e] * (dv[j][e] - dot);
            store_vec<Checked>(dxrow + 16 * vi, by, E::pack(yv[j]));
        }
    }
}

template <typename Tag, bool Checked>
__device__ __forceinline__ void row_bwd_smem(const unsigned char *sy, const unsigned char *sdy,
                                             unsigned char *dxrow, int nvec, int lane, const Bounds &by,
                                             const Bounds &bdy)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    float yv[EPV], dv[EPV], pr[EPV];
    uint4 ry, rd;
    float dot = 0.0f;
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(sy + 16 * vi, by, ry) || !load_vec<Checked>(sdy + 16 * vi, bdy, rd))
            continue;
        E::unpack(ry, yv);
        E::unpack(rd, dv);
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            pr[e] = yv[e] * dv[e];
        dot += tree_sum<EPV>(pr);
    }
    dot = group_sum<32>(dot);
    for (int vi = lane; vi < nvec; vi += 32) {
        if (!load_vec<Checked>(sy + 16 * vi, by, ry) || !load_vec<Checked>(sdy + 16 * vi, bdy, rd))
            continue;
        E::unpack(ry, yv);
        E::unpack(rd, dv);
#pragma unroll
        for (int e = 0; e < EPV; ++e)
            yv[e] = yv[e] * (dv[e] - dot);
        store_vec<Checked>(dxrow + 16 * vi, by, E::pack(yv));
    }
}

// Backward rows of a stage, dealt like consume_stage's: groups of G = 32/T
// rows round robin over the consumer warps from warp `first`.
template <typename Tag, bool Checked, int T, int V>
__device__ __forceinline__ int rows_bwd_registers(const unsigned char *sbuf, int half, const StageMeta &mt,
                                                  unsigned char *ybase, int row_bytes, int nvec, int first,
                                                  int lane, const Bounds &by, const Bounds &bdy)
{
    constexpr int G = 32 / T;
    const int g = lane / T, l = lane % T;
    for (int rb = first * G; rb < mt.nrows; rb += G * kConsumerWarps) {
        const int r = rb + g;
        row_bwd_registers<Tag, Checked, T, V>(sbuf + (size_t)r * row_bytes, sbuf + half + (size_t)r * row_bytes,
                                              ybase + (size_t)r * row_bytes, nvec, l, r < mt.nrows, by, bdy);
    }
    return (mt.nrows + G - 1) / G;
}

template <typename Tag, bool Checked>
__device__ __forceinline__ int consume_stage_bwd(const unsigned char *sbuf, int half, const StageMeta &mt,
                                                 unsigned char *y, int first, int lane, Bounds by)
{
    using E = Elem<Tag>;
    const int row_bytes = mt.C * E::kSize;
    const int nvec = row_bytes >> 4;
    unsigned char *ybase = y + mt.off * E::kSize;
    by.s_lo = sbuf;
    by.s_hi = sbuf + (size_t)mt.nrows * row_bytes;
    Bounds bdy = by;
    bdy.s_lo = sbuf + half;
    bdy.s_hi = sbuf + half + (size_t)mt.nrows * row_bytes;
    constexpr int VMAX = 16 / E::kPerVec;   // y and dy: at most 32 floats per lane
    if (nvec <= 8)
        return rows_bwd_registers<Tag, Checked, 8, 1>(sbuf, half, mt, ybase, row_bytes, nvec, first, lane, by,
                                                      bdy);
    if (nvec <= 16)
        return rows_bwd_registers<Tag, Checked, 8, 2>(sbuf, half, mt, ybase, row_bytes, nvec, first, lane, by,
                                                      bdy);
    if (nvec <= 32)
        return rows_bwd_registers<Tag, Checked, 16, 2>(sbuf, half, mt, ybase, row_bytes, nvec, first, lane, by,
                                                       bdy);
    if (nvec <= 64)
        return rows_bwd_registers<Tag, Checked, 32, 2>(sbuf, half, mt, ybase, row_bytes, nvec, first, lane, by,
                                                       bdy);
    if (VMAX >= 4 && nvec <= 128)
        return rows_bwd_registers<Tag, Checked, 32, (VMAX >= 4 ? 4 : 2)>(sbuf, half, mt, ybase, row_bytes, nvec,
                                                                         first, lane, by, bdy);
    for (int r = first; r < mt.nrows; r += kConsumerWarps)
        row_bwd_smem<Tag, Checked>(sbuf + (size_t)r * row_bytes, sbuf + half + (size_t)r * row_bytes,
                                   ybase + (size_t)r * row_bytes, nvec, lane, by, bdy);
    return mt.nrows;
}

// ------------------------------------------------------------ long rows
// A row longer than a stage is streamed through the stages twice, in
// chunks of equal length; all consumer warps share every chunk (warp w takes
// the vectors w*32 + lane, + 512, ...).  Pass 0 keeps a running (max m, sum s
// of exp(v - m)) per lane -- when the max grows, s is rescaled by exp(m_old -
// m_new) -- then the lanes, the warps (through shared memory) combine their
// pairs in a fixed order; pass 1 writes exp(v - m) / s.  For a whole row in
// one launch, pass 1 starts on the last chunk, still in its stage, and takes
// the others in reverse order.

// (m, s) of two partials; a -inf maximum contributes nothing.
__device__ __forceinline__ void combine_ms(float &m, float &s, float mo, float so)
{
    const float mn = fmaxf(m, mo);
    const float fa = m == mn ? 1.0f : ex2((m - mn) * kLog2e);
    const float fb = mo == mn ? 1.0f : ex2((mo - mn) * kLog2e);
    s = s * fa + so * fb;
    m = mn;
}

template <typename Tag, bool Checked>
__device__ __forceinline__ void long_chunk(const unsigned char *sbuf, const StageMeta &mt, unsigned char *y,
                                           bool causal, int warp, int lane, Bounds bd, float &m_l,
                                           float &s_l, float mL, float inv)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    const int nvec = (mt.C * E::kSize) >> 4;
    bd.s_lo = sbuf;
    bd.s_hi = sbuf + (size_t)mt.C * E::kSize;
    unsigned char *ybase = y + mt.off * E::kSize;
    const int row = mt.row0;
    for (int vi = warp * 32 + lane; vi < nvec; vi += kConsumerWarps * 32) {
        uint4 raw;
        if (!load_vec<Checked>(sbuf + 16 * vi, bd, raw))
            continue;
        float v[EPV];
        E::unpack(raw, v);
        const int col = mt.col0 + vi * EPV;
        const bool masked = causal && col > row;
        if (causal && !masked && col + EPV - 1 > row)
            apply_causal<EPV>(v, col, row);
        if (mt.pass == 0) {
            if (!masked) {
                const float vm = tree_max<EPV>(v);
                if (vm > m_l) {
                    s_l *= ex2((m_l - vm) * kLog2e);
                    m_l = vm;
                }
            }
            // while the running max is still -inf every value seen is -inf (or
            // NaN): it adds 0 (NaN), as a masked vector does; otherwise the
            // exponentials in fp32 pairs (the same bits as one at a time)
            if (masked || m_l == -INFINITY) {
                vec_exp<EPV>(v, m_l * kLog2e, true);
                s_l += tree_sum<EPV>(v);
            } else {
                s_l += vec_exp_sum_pairs<EPV>(v, m_l * kLog2e);
            }
        } else {
            vec_exp<EPV>(v, mL, masked);
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                v[e] *= inv;
            store_vec<Checked>(ybase + 16 * vi, bd, E::pack(v));
        }
    }
}

// Backward long rows: y and dy of a chunk sit in the two halves of a stage.
// Pass 0 adds this lane's y*dy products to dot_l (its vectors in order, chunk
// after chunk); pass 1 writes dx = y * (dy - dot).
template <typename Tag, bool Checked>
__device__ __forceinline__ void long_chunk_bwd(const unsigned char *sbuf, int half, const StageMeta &mt,
                                               unsigned char *dx, int warp, int lane, Bounds by, float &dot_l,
                                               float dot)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    const int nvec = (mt.C * E::kSize) >> 4;
    by.s_lo = sbuf;
    by.s_hi = sbuf + (size_t)mt.C * E::kSize;
    Bounds bdy = by;
    bdy.s_lo = sbuf + half;
    bdy.s_hi = sbuf + half + (size_t)mt.C * E::kSize;
    unsigned char *base = dx + mt.off * E::kSize;
    for (int vi = warp * 32 + lane; vi < nvec; vi += kConsumerWarps * 32) {
        uint4 ry, rd;
        if (!load_vec<Checked>(sbuf + 16 * vi, by, ry) || !load_vec<Checked>(sbuf + half + 16 * vi, bdy, rd))
            continue;
        float yv[EPV], dv[EPV];
        E::unpack(ry, yv);
        E::unpack(rd, dv);
        if (mt.pass == 0) {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                yv[e] *= dv[e];
            dot_l += tree_sum<EPV>(yv);
        } else {
#pragma unroll
            for (int e = 0; e < EPV; ++e)
                yv[e] = yv[e] * (dv[e] - dot);
            store_vec<Checked>(base + 16 * vi, by, E::pack(yv));
        }
    }
}

// The rows of a stage handled by one register routine: groups of T lanes,
// G = 32/T rows per group of a warp.  Row groups are dealt to the consumer
// warps round robin, starting at warp `first` (see consume_stage); q tracks
// each lane group's row inside its slice ((row0 + r) mod R) without a
// division per row.  Returns the number of row groups of the stage.
template <typename Tag, bool Checked, int T, int V>
__device__ __forceinline__ int rows_in_registers(const unsigned char *sbuf, const StageMeta &mt,
                                                 unsigned char *ybase, int row_bytes, int nvec,
                                                 bool causal, int first, int lane, const Bounds &bd)
{
    constexpr int G = 32 / T;
    const int g = lane / T, l = lane % T;
    const int step = G * kConsumerWarps;
    int q = 0, qstep = 0;
    if (causal) {
        q = (mt.row0 + first * G + g) % mt.R;
        qstep = step % mt.R;
    }
    const bool full_rows = nvec == T * V;
    for (int rb = first * G; rb < mt.nrows; rb += step) {
        const int r = rb + g;
        if constexpr (Elem<Tag>::kSize == 4)
            row_in_registers_scalar<Tag, Checked, T, V>(sbuf + (size_t)r * row_bytes,
                                                        ybase + (size_t)r * row_bytes, nvec, q, causal, l,
                                                        r < mt.nrows, bd);
        else if (full_rows && rb + G <= mt.nrows)   // warp-uniform
            row_in_registers_pairs<Tag, Checked, T, V, true>(sbuf + (size_t)r * row_bytes,
                                                             ybase + (size_t)r * row_bytes, nvec, q, causal, l,
                                                             true, bd);
        else
            row_in_registers_pairs<Tag, Checked, T, V, false>(sbuf + (size_t)r * row_bytes,
                                                              ybase + (size_t)r * row_bytes, nvec, q, causal, l,
                                                              r < mt.nrows, bd);
        q += qstep;
        if (q >= mt.R)
            q -= mt.R;
    }
    return (mt.nrows + G - 1) / G;
}

// All rows of one stage that belong to this consumer warp.  The routine
// depends on the row length only (see the table at the top of the file).
// Row groups are dealt round robin over the consumer warps starting at warp
// `first`; the caller advances `first` by the returned group count, so a
// stage with fewer groups than warps does not always land on the same warps.
template <typename Tag, bool Checked>
__device__ __forceinline__ int consume_stage(const unsigned char *sbuf, const StageMeta &mt,
                                             unsigned char *y, bool causal, int first, int lane,
                                             Bounds bd)
{
    using E = Elem<Tag>;
    const int row_bytes = mt.C * E::kSize;
    const int nvec = row_bytes >> 4;
    unsigned char *ybase = y + mt.off * E::kSize;
    bd.s_lo = sbuf;
    bd.s_hi = sbuf + (size_t)mt.nrows * row_bytes;
    if (nvec <= 8)
        return rows_in_registers<Tag, Checked, 8, 1>(sbuf, mt, ybase, row_bytes, nvec, causal, first, lane, bd);
    if (nvec <= 16)
        return rows_in_registers<Tag, Checked, 8, 2>(sbuf, mt, ybase, row_bytes, nvec, causal, first, lane, bd);
    if (nvec <= 32)
        return rows_in_registers<Tag, Checked, 8, 4>(sbuf, mt, ybase, row_bytes, nvec, causal, first, lane, bd);
    if (nvec <= 64)
        return rows_in_registers<Tag, Checked, 16, 4>(sbuf, mt, ybase, row_bytes, nvec, causal, first, lane,
                                                      bd);
    if (nvec <= 128)
        return rows_in_registers<Tag, Checked, 32, 4>(sbuf, mt, ybase, row_bytes, nvec, causal, first, lane,
                                                      bd);
    // one warp per row from here on
    int q = 0, qstep = 0;
    if (causal) {
        q = (mt.row0 + first) % mt.R;
        qstep = kConsumerWarps % mt.R;
    }
    for (int r = first; r < mt.nrows; r += kConsumerWarps) {
        const unsigned char *srow = sbuf + (size_t)r * row_bytes;
        unsigned char *yrow = ybase + (size_t)r * row_bytes;
        if constexpr (E::kSize == 4) {
            // fp32: rows up to 4 KiB in registers, longer ones in place in the stage
            if (nvec <= 256)
                row_in_registers_scalar<Tag, Checked, 32, 8>(srow, yrow, nvec, q, causal, lane, true, bd);
            else
                row_in_smem_inplace<Checked>(const_cast<unsigned char *>(srow), yrow, nvec, q, causal, lane,
                                             bd);
        } else {
            row_in_smem<Tag, Checked>(srow, yrow, nvec, q, causal, lane, bd);
        }
        q += qstep;
        if (q >= mt.R)
            q -= mt.R;
    }
    return mt.nrows;
}

// -------------------------------------------------------------- the schedule

// The pulling unit is a CTA, or for rows split over groups of CTAs a whole
// group (unit = group index, n_units = groups): the static and round-robin
// deals and the tail rule count units, not CTAs.
struct Puller {
    const KernelArgs &a;
    int32_t unit, n_units;
    int32_t k = 0;           // PULL_STATIC: patches taken so far
    int32_t slice = -1;      // PULL_RR_SLICE
    int32_t cur = 0, end = 0;
    int32_t q = 0;           // PULL_QUEUE: index into the try order
    int32_t die = 0;
    uint32_t fetch = kFetch; // PULL_QUEUE: patches per claim (1 near the end of a queue)

    __device__ explicit Puller(const KernelArgs &args)
        : Puller(args, static_cast<int32_t>(blockIdx.x), static_cast<int32_t>(gridDim.x))
    {
    }

    __device__ Puller(const KernelArgs &args, int32_t unit_, int32_t n_units_)
        : a(args), unit(unit_), n_units(n_units_)
    {
        if (a.mode == PULL_QUEUE && a.sm_die) {
            int d = a.sm_die[sm_id() & (BSM_MAX_SM - 1)];
            die = (d >= 0 && d < a.n_queues) ? d : 0;
        }
        // a short queue (small batch: about a patch per SM) is claimed one
        // patch at a time from the first claim on, so every SM gets one
        if (a.mode == PULL_QUEUE && static_cast<uint32_t>(a.queue_len[die]) < 2u * kFetch * static_cast<uint32_t>(n_units))
            fetch = 1;
        if (a.mode == PULL_RR_SLICE)
            slice = unit - n_units;
    }

    // Positions in a.items of this CTA's next patches (up to `most`, at most
    // kFetch); returns how many (0 when the CTA has no more work).
    __device__ int next_batch(int32_t (&pos)[kFetch], int most = kFetch)
    {
        int n = 0;
        if (a.mode == PULL_STATIC) {
#pragma unroll
            for (int j = 0; j < kFetch; ++j) {
                const int64_t idx = (int64_t)a.item_begin + unit + (int64_t)(k + j) * n_units;
                if (j < most && idx < a.item_end)
                    pos[n++] = static_cast<int32_t>(idx);
            }
            k += most;
            return n;
        }
        if (a.mode == PULL_RR_SLICE) {
            while (cur >= end) {
                slice += n_units;
                if (slice >= a.n_slices)
                    return 0;
                cur = a.slice_first_item[slice];
                end = a.slice_first_item[slice + 1];
            }
#pragma unroll
            for (int j = 0; j < kFetch; ++j)
                if (j < most && cur < end)
                    pos[n++] = cur++;
            return n;
        }
        // PULL_QUEUE: claim kFetch consecutive slots of the own die's queue,
        // then (steal) of the other dies' queues in order.
        const int tries = a.steal ? a.n_queues : 1;
        while (q < tries) {
            const int qq = (die + q) % a.n_queues;
            const uint32_t take = fetch < static_cast<uint32_t>(most) ? fetch : static_cast<uint32_t>(most);
            const uint32_t t = atomicAdd(&a.heads[qq], take);
            const uint32_t len = static_cast<uint32_t>(a.queue_len[qq]);
            if (t < len) {
#pragma unroll
                for (int j = 0; j < kFetch; ++j)
                    if (static_cast<uint32_t>(j) < take && t + j < len)
                        pos[n++] = a.queue_begin[qq] + static_cast<int32_t>(t + j);
                // near the end of the queue, claim one patch at a time so the
                // last patches spread over the SMs instead of queueing in fours
                if (len - t < 2u * kFetch * static_cast<uint32_t>(n_units))
                    fetch = 1;
                return n;
            }
            ++q;
        }
        return 0;
    }
};

// Warm L2 with the patches this CTA most likely copies first, before the
// wait on the previous kernel: the first kPrefetch slots of its first batch
// (the static deal's and round robin's exactly; under a queue, slots
// r*kFetch .. of queue u mod n_queues for CTA u = r*n_queues + (u mod
// n_queues), so that the CTAs together cover the first claims).  Two patches
// (19.5 MB over 152 SMs at 64 KiB) measured best: 1, 3 and 4 gave 0.4-0.7 %
// less on 384 x 512 x 512 rows, a second batch 2-5 % less (the prefetches
// then slow the previous kernel's last wave).  A prefetch into L2 carries no data to
// the SM and has no effect on what any load returns (L2 is the point of
// coherence), so it may run while the previous kernel still writes; what it
// buys is that DRAM serves these lines during that kernel's last wave
// instead of after it.  Records are checked like the producer checks them;
// one that fails is skipped.
constexpr int kPrefetch = 2;

__device__ __forceinline__ void prefetch_l2(const void *p, uint32_t bytes)
{
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

template <int ES>
__device__ __forceinline__ void prefetch_first_batch(const KernelArgs &a, bool two_inputs)
{
    int64_t first = 0, end = 0, step = 1;
    const int64_t u = blockIdx.x;
    if (a.mode == PULL_STATIC) {
        first = a.item_begin + u;
        end = a.item_end;
        step = gridDim.x;
    } else if (a.mode == PULL_RR_SLICE) {
        if (u >= a.n_slices)
            return;
        first = a.slice_first_item[u];
        end = a.slice_first_item[u + 1];
    } else {
        const int nq = a.n_queues > 0 ? a.n_queues : 1;
        const int q = static_cast<int>(u % nq);
        first = a.queue_begin[q] + (u / nq) * kFetch;
        end = (int64_t)a.queue_begin[q] + a.queue_len[q];
    }
    if (end > a.n_items)
        end = a.n_items;
    const int64_t cap = two_inputs ? a.stage_bytes / 2 : a.stage_bytes;
    for (int j = 0; j < kPrefetch; ++j) {
        const int64_t idx = first + j * step;
        if (idx < 0 || idx >= end)
            break;
        const Item it = a.items[idx];
        const int64_t ne = (int64_t)it.nrows * it.C;
        const int64_t nbytes = ne * ES;
        if (it.off < 0 || it.C <= 0 || it.nrows <= 0 || it.off + ne > a.total_elems || nbytes > cap ||
            (nbytes & 15) != 0 || ((it.off * ES) & 15) != 0)
            continue;
        prefetch_l2(static_cast<const unsigned char *>(a.x) + it.off * ES, static_cast<uint32_t>(nbytes));
        if (two_inputs)
            prefetch_l2(static_cast<const unsigned char *>(a.x2) + it.off * ES, static_cast<uint32_t>(nbytes));
    }
}

template <typename Tag, int Op, bool Checked>
__global__ void __launch_bounds__(kThreads, 1) softmax_persistent(const KernelArgs a)
{
    using E = Elem<Tag>;
    // the long-row machinery is compiled into its own instance, so plans
    // without long rows do not pay its registers
    constexpr bool kLong = Op == OP_FORWARD_LONG || Op == OP_BACKWARD_LONG;
    constexpr bool kBwd = Op == OP_BACKWARD || Op == OP_BACKWARD_LONG;
    extern __shared__ __align__(1024) unsigned char smem[];
    SmemHeader &h = *reinterpret_cast<SmemHeader *>(smem);
    unsigned char *stages = smem + kSmemHeader;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = a.n_stages;
    const uint64_t wait_limit = a.wait_limit_ns ? a.wait_limit_ns : kWaitLimitNs;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&h.full[s], 1);
            mbar_init(&h.empty[s], kConsumerWarps);
        }
        mbar_init(&h.xwarp, kConsumerWarps);
        h.abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    // rows that fit a stage: the first batch's bytes are prefetched into L2
    // (a hint: it reads nothing into this CTA and writes nothing)
    if (!kLong && warp == kConsumerWarps && lane == 0)
        prefetch_first_batch<E::kSize>(a, kBwd);
    // Programmatic dependent launch: this kernel may have started while the
    // previous kernel of the stream was finishing.  No role loads data,
    // stores or starts a bounded wait before that kernel is done (a no-op
    // without such a predecessor); then the next kernel may begin its own
    // launch.
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");

    if (warp == kConsumerWarps) {
        // ------------------------------------------------------- producer
        if (lane == 0) {
            Puller pull(a);
            uint32_t issued_phase[kMaxStages];
            bool issued[kMaxStages];
            for (int s = 0; s < kMaxStages; ++s)
                issued[s] = false;
            bool aborted = false, done = false;
            uint32_t it = 0;
            // take the next stage of the ring once the consumers released it
            auto next_stage = [&](int &s, uint32_t &ph) -> bool {
                s = static_cast<int>(it % S);
                ph = (it / S) & 1u;
                if (!mbar_wait_bounded(&h.empty[s], ph ^ 1u, &h.abort_flag, wait_limit)) {
                    aborted = true;
                    return false;
                }
                issued[s] = false;
                ++it;
                return true;
            };
            // Long-row instances claim one patch at a time, and the next one
            // while a row streams: the queue atomic and the record loads
            // behind it are round trips of microseconds under full load,
            // which would otherwise stall the ring at every row start.
            int nx_n = -1;              // patches claimed ahead (-1: none)
            int32_t nx_pos = 0;
            Item nx_item{0, 0, 0, 0, 0};
            LongSeg nx_seg{0, 0, 0, 0};
            auto claim_ahead = [&]() {
                int32_t p1[kFetch];
                nx_n = pull.next_batch(p1, 1);
                nx_pos = p1[0];
                if (nx_n > 0 && nx_pos >= 0 && nx_pos < a.n_items) {
                    nx_item = a.items[nx_pos];
                    nx_seg = a.segs ? a.segs[nx_pos] : LongSeg{0, 0, 0, 0};
                }
            };
            while (!done && !aborted) {
                // the next patches: their records load in parallel
                int32_t pos[kFetch];
                Item batch[kFetch];
                LongSeg lseg[kFetch];   // long-row instances: the segment records
                int n = 0;
                if (kLong && nx_n >= 0) {
                    n = nx_n;
                    pos[0] = nx_pos;
                    batch[0] = nx_item;
                    lseg[0] = nx_seg;
                    nx_n = -1;
                } else {
                    n = pull.next_batch(pos, kLong ? 1 : kFetch);
#pragma unroll
                    for (int j = 0; j < kFetch; ++j)
                        if (j < n && pos[j] >= 0 && pos[j] < a.n_items) {
                            batch[j] = a.items[pos[j]];
                            if (kLong && a.segs)
                                lseg[j] = a.segs[pos[j]];
                        }
                }
                if (n == 0) {
                    // no more work: tell the consumers through the next stage
                    int s = 0;
                    uint32_t ph = 0;
                    if (!next_stage(s, ph))
                        break;
                    h.meta[s].kind = KIND_DONE;
                    mbar_arrive(&h.full[s]);
                    done = true;
                    break;
                }
                for (int j = 0; j < n && !aborted; ++j) {
                    // long-row instances check the patch (and cut a long one
                    // into chunks) before the wait for its stage, the others
                    // after it
                    int s = 0;
                    uint32_t ph = 0;
                    if (!kLong && !next_stage(s, ph))
                        break;
                    const Item item = batch[j];
                    const int64_t ne = (int64_t)item.nrows * item.C;
                    const int64_t nbytes = ne * E::kSize;
                    const int64_t cap = kBwd ? a.stage_bytes / 2 : a.stage_bytes;
                    LongSeg sg{0, 0, 0, 0};
                    if (kLong && a.segs && pos[j] >= 0 && pos[j] < a.n_items)
                        sg = lseg[j];
                    const bool is_long = kLong && sg.part_count > 0;
                    const bool ok = pos[j] >= 0 && pos[j] < a.n_items && item.off >= 0 && item.C > 0 &&
                                    item.nrows > 0 && item.R > 0 && item.row0 >= 0 &&
                                    item.row0 < item.R && item.off + ne <= a.total_elems &&
                                    (nbytes <= cap || is_long) && (nbytes & 15) == 0 &&
                                    ((item.off * E::kSize) & 15) == 0 && (!is_long || item.nrows == 1) &&
                                    (!is_long || (sg.part >= sg.part_first &&
                                                  sg.part < sg.part_first + sg.part_count && sg.part_first >= 0));
                    // a long segment: chunks of equal length in whole 16-byte
                    // vectors (no short last chunk leaves the consumers waiting
                    // on the next copy), every one non-empty; 32-bit arithmetic
                    // (C < 2^31, a stage < 2^18 bytes)
                    int64_t chunk = 1, nch = 0;
                    if (kLong && is_long && ok) {
                        const uint32_t cl = static_cast<uint32_t>(item.C);
                        const uint32_t cmax = static_cast<uint32_t>(cap / E::kSize);
                        const uint32_t n_min = (cl + cmax - 1) / cmax;
                        const uint32_t c = ((cl + n_min - 1) / n_min + E::kPerVec - 1) & ~uint32_t(E::kPerVec - 1);
                        chunk = c;
                        nch = (cl + c - 1) / c;
                    }
                    if (kLong && !next_stage(s, ph))
                        break;
                    StageMeta &mt = h.meta[s];
                    if ((a.debug & KDEBUG_WITHHOLD_STAGE0) && it == 1)
                        continue;                      // test hook: stage 0 is never filled
                    if (!ok) {
                        atomicOr(a.status, BSM_DEV_BOUNDS);
                        mt.kind = KIND_SKIP;
                        mbar_arrive(&h.full[s]);
                        continue;
                    }
                    if (kLong && is_long) {
                        // the segment in chunks of one stage: a whole row (one
                        // segment) streams twice in this launch; a segment of a
                        // longer row streams once, for this launch's phase
                        // a whole row with fewer chunks than stages stays staged:
                        // its second pass needs no copies
                        const bool resident = sg.part_count == 1 && nch < S;
                        const int p_lo = sg.part_count == 1 ? 0 : a.phase;
                        const int p_hi = sg.part_count == 1 && !resident ? 1 : a.phase;
                        bool first_stage = true;
                        for (int pass = p_lo; pass <= p_hi && !aborted; ++pass) {
                        // a whole row's second pass runs backwards from its
                        // last chunk, which the consumers keep in its stage
                        // and finish first (no copy); the others follow, the
                        // most recently read (most likely still in L2) first
                        const bool rev = pass == 1 && sg.part_count == 1;
                        for (int64_t kk = 0; kk < (rev ? nch - 1 : nch) && !aborted; ++kk) {
                            const int64_t k = rev ? nch - 2 - kk : kk;
                            if (!first_stage && !next_stage(s, ph))
                                break;
                            first_stage = false;
                            StageMeta &lm = h.meta[s];
                            const int64_t c0 = k * chunk;
                            const int64_t cn = item.C - c0 < chunk ? item.C - c0 : chunk;
                            lm.off = item.off + c0;
                            lm.C = static_cast<int32_t>(cn);
                            lm.nrows = 1;
                            lm.row0 = item.row0;
                            lm.R = item.R;
                            lm.col0 = static_cast<int32_t>(sg.col0 + c0);
                            lm.pass = pass;
                            lm.last = rev ? k == 0 : k == nch - 1;
                            lm.first = rev ? kk == 0 : k == 0;
                            lm.part = sg.part;
                            lm.part_first = sg.part_first;
                            lm.part_count = sg.part_count;
                            lm.resident = resident;
                            lm.kind = KIND_LONG;
                            const uint32_t cb = static_cast<uint32_t>(cn * E::kSize);
                            unsigned char *ldst = stages + (size_t)s * a.stage_bytes;
                            mbar_arrive_expect_tx(&h.full[s], kBwd ? 2 * cb : cb);
                            bulk_load(ldst,
                                      static_cast<const unsigned char *>(a.x) + (item.off + c0) * E::kSize,
                                      cb, &h.full[s]);
                            if (kBwd)   // dy's chunk into the second half
                                bulk_load(ldst + a.stage_bytes / 2,
                                          static_cast<const unsigned char *>(a.x2) + (item.off + c0) * E::kSize,
                                          cb, &h.full[s]);
                            issued[s] = true;
                            issued_phase[s] = ph;
                            // the row's second chunk is on its way (or its only
                            // one): claim the next patch now
                            if (nx_n < 0 && j == n - 1 && pass == p_lo && (kk == 1 || nch == 1))
                                claim_ahead();
                        }
                        }
                        continue;
                    }
                    mt.off = item.off;
                    mt.C = item.C;
                    mt.nrows = item.nrows;
                    mt.row0 = item.row0;
                    mt.R = item.R;
                    mt.kind = KIND_DATA;
                    const uint32_t bytes = static_cast<uint32_t>(nbytes);
                    unsigned char *dst = stages + (size_t)s * a.stage_bytes;
                    const unsigned char *src = static_cast<const unsigned char *>(a.x) + item.off * E::kSize;
                    const int half = a.stage_bytes / 2;
                    const unsigned char *src2 =
                        kBwd ? static_cast<const unsigned char *>(a.x2) + item.off * E::kSize : nullptr;
                    if (Checked) {
                        const unsigned char *x0 = static_cast<const unsigned char *>(a.x);
                        bool bad = s < 0 || s >= S || S > kMaxStages ||
                                   src < x0 || src + bytes > x0 + a.total_elems * E::kSize ||
                                   (reinterpret_cast<uintptr_t>(src) & 15) ||
                                   (smem_addr(dst) & 15) || (bytes & 15) || bytes == 0 ||
                                   dst + bytes > smem + kSmemHeader + (size_t)S * a.stage_bytes;
                        if (kBwd) {
                            const unsigned char *g0 = static_cast<const unsigned char *>(a.x2);
                            bad = bad || bytes > (uint32_t)half || src2 < g0 ||
                                  src2 + bytes > g0 + a.total_elems * E::kSize ||
                                  (reinterpret_cast<uintptr_t>(src2) & 15) || (half & 15);
                        }
                        if (bad) {
                            check_fail(a.status, 3, static_cast<uint64_t>(pos[j]), bytes);
                            mt.kind = KIND_SKIP;
                            mbar_arrive(&h.full[s]);
                            continue;
                        }
                    }
                    if (kBwd) {
                        mbar_arrive_expect_tx(&h.full[s], 2 * bytes);
                        bulk_load(dst, src, bytes, &h.full[s]);
                        bulk_load(dst + half, src2, bytes, &h.full[s]);
                    } else {
                        mbar_arrive_expect_tx(&h.full[s], bytes);
                        bulk_load(dst, src, bytes, &h.full[s]);
                    }
                    issued[s] = true;
                    issued_phase[s] = ph;
                }
            }
            if (aborted) {
                atomicOr(a.status, BSM_DEV_TIMEOUT);
                h.abort_flag = 1;
            }
            // every copy this lane issued has landed before it leaves (normally
            // they have: the consumers waited for them; after an abort they may not)
            for (int s = 0; s < S; ++s)
                if (issued[s])
                    mbar_wait_bounded(&h.full[s], issued_phase[s], nullptr, wait_limit);
            if (a.mode == PULL_QUEUE) {
                // the last CTA to finish pulling rewinds the queue heads
                __threadfence();
                const uint32_t prev = atomicAdd(&a.heads[BSM_MAX_DIES], 1u);
                if (prev == gridDim.x - 1) {
                    for (int d = 0; d < BSM_MAX_DIES; ++d)
                        atomicExch(&a.heads[d], 0u);
                    atomicExch(&a.heads[BSM_MAX_DIES], 0u);
                }
            }
        }
        return;
    }

    // ----------------------------------------------------------- consumers
    const bool causal = (a.flags & BSM_FLAG_CAUSAL) != 0;
    unsigned char *y = static_cast<unsigned char *>(a.y);
    uint32_t groups_seen = 0;   // row groups dealt so far (the same count in every warp)
    // long rows: this lane's running (max, sum); the row's final exponent
    // offset and reciprocal; which partial buffer and barrier phase is next
    float m_l = -INFINITY, s_l = 0.0f, long_mL = 0.0f, long_inv = 0.0f;
    uint32_t long_rows = 0;
    uint32_t long_first_it = 0;  // stage iteration of the current row's first chunk
    (void)m_l, (void)s_l, (void)long_mL, (void)long_inv, (void)long_rows;
    for (uint32_t it = 0;; ++it) {
        const int s = it % S;
        const uint32_t ph = (it / S) & 1u;
        if (!mbar_wait_bounded(&h.full[s], ph, &h.abort_flag, wait_limit)) {
            if (lane == 0) {
                atomicOr(a.status, BSM_DEV_TIMEOUT);
                h.abort_flag = 1;
            }
            break;
        }
        const StageMeta mt = h.meta[s];
        if (mt.kind == KIND_DONE)
            break;
        if (kLong && mt.kind == KIND_LONG) {
            Bounds bd{nullptr, nullptr, y, y + a.total_elems * E::kSize, a.status};
            if (mt.pass == 1 && mt.first && mt.part_count > 1) {
                // the row's partials, left by phase 0, combined in slot order
                // (every segment of the row, on any SM, gets the same result)
                const float *pp = a.partials + 2 * static_cast<int64_t>(mt.part_first);
                if constexpr (kBwd) {
                    float dot = 0.0f;
                    for (int k = 0; k < mt.part_count; ++k)
                        dot += pp[2 * k];
                    long_mL = dot;
                } else {
                    float m = -INFINITY, sum = 0.0f;
                    for (int k = 0; k < mt.part_count; ++k)
                        combine_ms(m, sum, pp[2 * k], pp[2 * k + 1]);
                    long_mL = m * kLog2e;
                    long_inv = __frcp_rn(sum);
                }
            }
            if constexpr (kBwd)
                long_chunk_bwd<Tag, Checked>(stages + (size_t)s * a.stage_bytes, a.stage_bytes / 2, mt, y, warp,
                                             lane, bd, s_l, long_mL);
            else
                long_chunk<Tag, Checked>(stages + (size_t)s * a.stage_bytes, mt, y, causal, warp, lane, bd, m_l,
                                         s_l, long_mL, long_inv);
            __syncwarp();
            if (mt.pass == 0 && mt.first)
                long_first_it = it;
            // a whole row keeps its last chunk (a resident row: every chunk)
            // staged for the second pass
            const bool keep = mt.resident || (mt.pass == 0 && mt.last && mt.part_count == 1);
            if (lane == 0 && !keep)
                mbar_arrive(&h.empty[s]);
            if (mt.pass == 0 && mt.last) {
                // the segment's partial: lanes, then warps in a fixed order
                if constexpr (kBwd) {
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1)
                        s_l += __shfl_xor_sync(0xFFFFFFFFu, s_l, o);
                } else {
#pragma unroll
                    for (int o = 16; o >= 1; o >>= 1) {
                        const float mo = __shfl_xor_sync(0xFFFFFFFFu, m_l, o);
                        const float so = __shfl_xor_sync(0xFFFFFFFFu, s_l, o);
                        combine_ms(m_l, s_l, mo, so);
                    }
                }
                const int par = long_rows & 1;
                if (lane == 0) {
                    h.partial[par][warp] = make_float2(kBwd ? s_l : m_l, kBwd ? 0.0f : s_l);
                    mbar_arrive(&h.xwarp);
                }
                if (!mbar_wait_bounded(&h.xwarp, long_rows & 1u, &h.abort_flag, wait_limit)) {
                    if (lane == 0) {
                        atomicOr(a.status, BSM_DEV_TIMEOUT);
                        h.abort_flag = 1;
                    }
                    break;
                }
                float m = -INFINITY, sum = 0.0f;
                for (int w = 0; w < kConsumerWarps; ++w) {
                    const float2 pw = h.partial[par][w];
                    if constexpr (kBwd)
                        m = w == 0 ? pw.x : m + pw.x;
                    else
                        combine_ms(m, sum, pw.x, pw.y);
                }
                if (mt.part_count == 1) {
                    // the whole row: its second pass follows in this launch,
                    // starting on the chunk still in this stage
                    if constexpr (kBwd) {
                        long_mL = m;
                    } else {
                        long_mL = m * kLog2e;
                        long_inv = __frcp_rn(sum);
                    }
                    if (!mt.resident) {
                        StageMeta m1 = mt;
                        m1.pass = 1;
                        if constexpr (kBwd)
                            long_chunk_bwd<Tag, Checked>(stages + (size_t)s * a.stage_bytes, a.stage_bytes / 2, m1,
                                                         y, warp, lane, bd, s_l, long_mL);
                        else
                            long_chunk<Tag, Checked>(stages + (size_t)s * a.stage_bytes, m1, y, causal, warp, lane,
                                                     bd, m_l, s_l, long_mL, long_inv);
                        __syncwarp();
                        if (lane == 0)
                            mbar_arrive(&h.empty[s]);
                    } else {
                        // a resident row: every chunk, from the first one's stage
                        for (uint32_t j = long_first_it; j <= it; ++j) {
                            const int sj = static_cast<int>(j % S);
                            StageMeta m1 = h.meta[sj];
                            m1.pass = 1;
                            if constexpr (kBwd)
                                long_chunk_bwd<Tag, Checked>(stages + (size_t)sj * a.stage_bytes,
                                                             a.stage_bytes / 2, m1, y, warp, lane, bd, s_l, long_mL);
                            else
                                long_chunk<Tag, Checked>(stages + (size_t)sj * a.stage_bytes, m1, y, causal, warp,
                                                         lane, bd, m_l, s_l, long_mL, long_inv);
                        }
                        __syncwarp();
                        if (lane == 0)
                            for (uint32_t j = long_first_it; j <= it; ++j)
                                mbar_arrive(&h.empty[j % S]);
                    }
                } else if (warp == 0 && lane == 0) {
                    a.partials[2 * static_cast<int64_t>(mt.part)] = m;
                    a.partials[2 * static_cast<int64_t>(mt.part) + 1] = sum;
                }
                m_l = -INFINITY;
                s_l = 0.0f;
                ++long_rows;
            }
            continue;
        }
        if (mt.kind == KIND_DATA) {
            Bounds bd{nullptr, nullptr, y, y + a.total_elems * E::kSize, a.status};
            const int64_t cap = kBwd ? a.stage_bytes / 2 : a.stage_bytes;
            if (Checked && (mt.nrows <= 0 || mt.C <= 0 || (int64_t)mt.nrows * mt.C * E::kSize > cap)) {
                if (lane == 0)
                    check_fail(a.status, 4, static_cast<uint64_t>(mt.nrows), static_cast<uint64_t>(mt.C));
            } else {
                const int first = static_cast<int>((warp + kConsumerWarps - groups_seen % kConsumerWarps) %
                                                   kConsumerWarps);
                if constexpr (kBwd)
                    groups_seen += consume_stage_bwd<Tag, Checked>(stages + (size_t)s * a.stage_bytes,
                                                                   a.stage_bytes / 2, mt, y, first, lane, bd);
                else
                    groups_seen += consume_stage<Tag, Checked>(stages + (size_t)s * a.stage_bytes, mt, y,
                                                               causal, first, lane, bd);
            }
        }
        __syncwarp();
        if (lane == 0)
            mbar_arrive(&h.empty[s]);
    }
}


// ------------------------------------------------ rows over groups of CTAs
// A row too long for one SM's shared memory is cut into K parts of equal
// length (whole 16-byte vectors; the last may be shorter or empty), and the K
// CTAs of a group each stage one part in one stage: every element is read
// from memory once.  Each CTA takes its part's running (max, rescaled sum)
// -- threads, then warps in a fixed order -- and publishes it in global
// memory as two words tagged with the row's sequence number; every member
// then reads the K partials until all carry the tag, combines them in the
// same fixed order (a per-lane sum over ranks l, l + 32, ..., then the xor
// tree), and writes its part of y.  The consumers work one row ahead: they
// take the next row's partial (from its stage) before finishing the previous
// row (held in registers), so the exchange overlaps work.  The group's
// rank-0 CTA claims the rows (any policy's puller, with the group as the
// unit) and announces them to its members through a ring of claim words.
// The launch is cooperative, so every member of a group is resident and each
// wait ends; every wait is bounded all the same.

__device__ __forceinline__ void st_release_u64(unsigned long long *p, unsigned long long v)
{
    asm volatile("st.release.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ void st_relaxed_u64(unsigned long long *p, unsigned long long v)
{
    asm volatile("st.relaxed.gpu.global.u64 [%0], %1;" ::"l"(p), "l"(v) : "memory");
}

__device__ __forceinline__ unsigned long long ld_acquire_u64(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.acquire.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ unsigned long long ld_relaxed_u64(const unsigned long long *p)
{
    unsigned long long v;
    asm volatile("ld.relaxed.gpu.global.u64 %0, [%1];" : "=l"(v) : "l"(p) : "memory");
    return v;
}

// Wait until the claim word at p carries sequence number seq (bounded).
__device__ __noinline__ bool wait_claim(const unsigned long long *p, uint32_t seq, const volatile int32_t *abort,
                                        uint64_t limit_ns, unsigned long long &word)
{
    word = ld_acquire_u64(p);
    if (static_cast<uint32_t>(word >> 32) == seq)
        return true;
    const uint64_t t0 = global_timer_ns();
    for (uint32_t it = 0; it < (1u << 26); ++it) {
        __nanosleep(32);
        word = ld_acquire_u64(p);
        if (static_cast<uint32_t>(word >> 32) == seq)
            return true;
        if ((abort && *abort) || global_timer_ns() - t0 > limit_ns)
            return false;
    }
    return false;
}

__device__ __forceinline__ unsigned long long pack_ms(float m, float sum)
{
    return (static_cast<unsigned long long>(__float_as_uint(sum)) << 32) | __float_as_uint(m);
}

// A member's part of a group row held in registers: consumer thread t (of
// the kConsumerWarps * 32) holds the part's 16-byte vectors t, t + 512, ...
constexpr int kConsumerThreads = kConsumerWarps * 32;

template <typename Tag, bool Checked>
__device__ __forceinline__ void group_load(uint4 (&r)[kGroupVecs], const unsigned char *sbuf, int nvec, int tid,
                                           const Bounds &bd)
{
    using E = Elem<Tag>;
#pragma unroll
    for (int j = 0; j < kGroupVecs; ++j) {
        const int vi = tid + j * kConsumerThreads;
        r[j] = E::neg_inf_vec();
        if (vi < nvec) {
            uint4 t;
            if (load_vec<Checked>(sbuf + 16 * vi, bd, t))
                r[j] = t;
        }
    }
}

// This thread's running (max, sum of exp(v - max)) over its vectors of the
// part in the stage, in chunks of 16 elements (4 fp32 or 2 bf16 vectors, so
// the chunk's unpacked values and the held row fit the registers): a chunk's vectors are
// loaded first (independent loads), then its maximum taken (bf16 without
// the causal mask: on the packed words) and, when it grows the running one,
// the sum rescaled; then the chunk's exponentials added in vector order,
// computed in fp32 pairs (the same bits as one at a time: each pair is two
// IEEE operations, each vector's sum in tree_sum's order).  While the
// running maximum is -inf every value seen is -inf (masked) or NaN: it adds
// 0 (NaN).  `mid` runs halfway through (the
// caller issues its exchange loads there).
template <typename Tag, bool Checked, typename Mid>
__device__ __forceinline__ void group_partial(const unsigned char *sbuf, int nvec, int tid, int col0, int row,
                                              bool causal, const Bounds &bd, float &m, float &s, Mid &&mid)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    constexpr int kGroupChunk = 16 / EPV;
    m = -INFINITY;
    s = 0.0f;
#pragma unroll
    for (int c = 0; c < kGroupVecs; c += kGroupChunk) {
        if (c == kGroupVecs / 2)
            mid();
        uint4 raw[kGroupChunk];
#pragma unroll
        for (int j = 0; j < kGroupChunk; ++j) {
            const int vi = tid + (c + j) * kConsumerThreads;
            raw[j] = E::neg_inf_vec();
            if (vi < nvec) {
                uint4 t;
                if (load_vec<Checked>(sbuf + 16 * vi, bd, t))
                    raw[j] = t;
            }
        }
        float cm = -INFINITY;
        float v[kGroupChunk][EPV];
        if (causal) {
#pragma unroll
            for (int j = 0; j < kGroupChunk; ++j) {
                const int col = col0 + (tid + (c + j) * kConsumerThreads) * EPV;
                E::unpack(raw[j], v[j]);
                if (col + EPV - 1 > row)
                    apply_causal<EPV>(v[j], col, row);
                cm = fmaxf(cm, tree_max<EPV>(v[j]));
            }
        } else {
#pragma unroll
            for (int j = 0; j < kGroupChunk; ++j)
                E::unpack(raw[j], v[j]);
            cm = raw_max<Tag, kGroupChunk>(raw, v);
        }
        if (cm > m) {
            s *= ex2((m - cm) * kLog2e);
            m = cm;
        }
        const float mL = m * kLog2e;
#pragma unroll
        for (int j = 0; j < kGroupChunk; ++j) {
            const int vi = tid + (c + j) * kConsumerThreads;
            const int col = col0 + vi * EPV;
            if (vi < nvec) {
                if ((causal && col > row) || m == -INFINITY) {
                    vec_exp<EPV>(v[j], mL, true);
                    s += tree_sum<EPV>(v[j]);
                } else {
                    s += vec_exp_sum_pairs<EPV>(v[j], mL);
                }
            }
        }
    }
}

// y = exp(v - M) / S for this thread's vectors of the part (mL = M log2 e),
// in fp32 pairs where no element is masked.
template <typename Tag, bool Checked>
__device__ __forceinline__ void group_write(const uint4 (&r)[kGroupVecs], int nvec, int tid, int col0, int row,
                                            bool causal, float mL, float inv, unsigned char *ypart, const Bounds &bd)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
#pragma unroll
    for (int j = 0; j < kGroupVecs; ++j) {
        const int vi = tid + j * kConsumerThreads;
        if (vi < nvec) {
            const int col = col0 + vi * EPV;
            const bool masked = causal && col > row;
            float v[EPV];
            E::unpack(r[j], v);
            if (causal && !masked && col + EPV - 1 > row)
                apply_causal<EPV>(v, col, row);
            if (masked) {
                vec_exp<EPV>(v, mL, true);
#pragma unroll
                for (int e = 0; e < EPV; ++e)
                    v[e] *= inv;
            } else {
                const float2 l2 = make_float2(kLog2e, kLog2e), nm = make_float2(-mL, -mL);
                const float2 i2 = make_float2(inv, inv);
#pragma unroll
                for (int e = 0; e < EPV; e += 2) {
                    const float2 t = fma2(make_float2(v[e], v[e + 1]), l2, nm);
                    const float2 y2 = mul2(make_float2(ex2(t.x), ex2(t.y)), i2);
                    v[e] = y2.x;
                    v[e + 1] = y2.y;
                }
            }
            store_vec<Checked>(ypart + 16 * vi, bd, E::pack(v));
        }
    }
}

template <typename Tag, bool Checked>
__global__ void __launch_bounds__(kThreads, 1) softmax_group(const KernelArgs a)
{
    using E = Elem<Tag>;
    constexpr int EPV = E::kPerVec;
    extern __shared__ __align__(1024) unsigned char smem[];
    SmemHeader &h = *reinterpret_cast<SmemHeader *>(smem);
    unsigned char *stages = smem + kSmemHeader;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = a.n_stages;
    const int K = a.group_k;
    const int grp = static_cast<int>(blockIdx.x) / K, rank = static_cast<int>(blockIdx.x) % K;
    const uint64_t wait_limit = a.wait_limit_ns ? a.wait_limit_ns : kWaitLimitNs;
    unsigned long long *ring = a.ring + static_cast<size_t>(grp) * kGroupRing;
    unsigned long long *xch = a.xch + 2 * static_cast<size_t>(grp) * kGroupSlots * K;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&h.full[s], 1);
            mbar_init(&h.empty[s], kConsumerWarps);
        }
        h.xarrive[0] = h.xarrive[1] = 0u;
        h.abort_flag = 0;
        mbar_init_fence();
    }
    __syncthreads();
    asm volatile("griddepcontrol.wait;" ::: "memory");

    if (warp == kConsumerWarps) {
        // ------------------------------------------------------- producer
        if (lane == 0) {
            Puller pull(a, grp, a.n_groups);
            uint32_t issued_phase[kMaxStages];
            bool issued[kMaxStages];
            for (int s = 0; s < kMaxStages; ++s)
                issued[s] = false;
            bool aborted = false;
            uint32_t it = 0, posted = 0;
            bool post_done = false;
            for (uint32_t t = 0; !aborted; ++t) {
                if (rank == 0) {
                    // announce rows up to kClaimAhead beyond this one
                    while (!post_done && posted <= t + kClaimAhead) {
                        int32_t p1[kFetch];
                        const int n = pull.next_batch(p1, 1);
                        const uint32_t pos = n > 0 ? static_cast<uint32_t>(p1[0]) : 0xFFFFFFFFu;
                        st_release_u64(&ring[posted % kGroupRing],
                                       (static_cast<unsigned long long>(posted + 1) << 32) | pos);
                        ++posted;
                        post_done = n == 0;
                    }
                }
                unsigned long long word = 0;
                if (!wait_claim(&ring[t % kGroupRing], t + 1, &h.abort_flag, wait_limit, word)) {
                    aborted = true;
                    break;
                }
                const uint32_t pos = static_cast<uint32_t>(word);
                const int s = static_cast<int>(it % S);
                const uint32_t ph = (it / S) & 1u;
                if (!mbar_wait_bounded(&h.empty[s], ph ^ 1u, &h.abort_flag, wait_limit)) {
                    aborted = true;
                    break;
                }
                issued[s] = false;
                ++it;
                StageMeta &mt = h.meta[s];
                if (pos == 0xFFFFFFFFu) {
                    mt.kind = KIND_DONE;
                    mbar_arrive(&h.full[s]);
                    break;
                }
                if ((a.debug & KDEBUG_WITHHOLD_STAGE0) && it == 1)
                    continue;                      // test hook: stage 0 is never filled
                const bool in = pos < static_cast<uint32_t>(a.n_items);
                const Item item = in ? a.items[pos] : Item{-1, 0, 0, 0, 0};
                // this member's part (the same cut in every member)
                const int64_t part = ((int64_t(item.C) + K - 1) / K + EPV - 1) / EPV * EPV;
                const int64_t c0 = part * rank;
                const int64_t cn = item.C - c0 < 0 ? 0 : (item.C - c0 < part ? item.C - c0 : part);
                const bool ok = in && item.off >= 0 && item.C > 0 && item.nrows == 1 && item.R > 0 &&
                                item.row0 >= 0 && item.row0 < item.R && item.off + item.C <= a.total_elems &&
                                ((item.off * E::kSize) & 15) == 0 && ((int64_t(item.C) * E::kSize) & 15) == 0 &&
                                part * E::kSize <= a.stage_bytes &&
                                part * E::kSize <= int64_t(kGroupVecs) * 16 * kConsumerThreads;
                if (!ok) {
                    // every member sees the same record and skips the row alike
                    atomicOr(a.status, BSM_DEV_BOUNDS);
                    mt.kind = KIND_SKIP;
                    mbar_arrive(&h.full[s]);
                    continue;
                }
                mt.off = item.off + c0;
                mt.C = static_cast<int32_t>(cn);
                mt.nrows = 1;
                mt.row0 = item.row0;
                mt.R = item.R;
                mt.col0 = static_cast<int32_t>(c0);
                mt.pass = 0;
                mt.kind = KIND_GROUP;
                if (cn == 0) {
                    mbar_arrive(&h.full[s]);
                    continue;
                }
                const uint32_t bytes = static_cast<uint32_t>(cn * E::kSize);
                unsigned char *dst = stages + static_cast<size_t>(s) * a.stage_bytes;
                const unsigned char *src = static_cast<const unsigned char *>(a.x) + (item.off + c0) * E::kSize;
                if (Checked) {
                    const unsigned char *x0 = static_cast<const unsigned char *>(a.x);
                    if (src < x0 || src + bytes > x0 + a.total_elems * E::kSize ||
                        (reinterpret_cast<uintptr_t>(src) & 15) || (smem_addr(dst) & 15) ||
                        bytes > static_cast<uint32_t>(a.stage_bytes) ||
                        dst + bytes > smem + kSmemHeader + static_cast<size_t>(S) * a.stage_bytes) {
                        check_fail(a.status, 3, pos, bytes);
                        mt.kind = KIND_SKIP;       // the group's other members time out
                        mbar_arrive(&h.full[s]);
                        continue;
                    }
                }
                mbar_arrive_expect_tx(&h.full[s], bytes);
                bulk_load(dst, src, bytes, &h.full[s]);
                issued[s] = true;
                issued_phase[s] = ph;
            }
            if (aborted) {
                atomicOr(a.status, BSM_DEV_TIMEOUT);
                h.abort_flag = 1;
            }
            for (int s = 0; s < S; ++s)
                if (issued[s])
                    mbar_wait_bounded(&h.full[s], issued_phase[s], nullptr, wait_limit);
        }
        __syncwarp();
    } else {
        // ----------------------------------------------------------- consumers
        // A member takes a row's partial straight from its stage, then writes
        // the previous row -- held in registers (thread t of the 512 consumer
        // threads holds its vectors t, t + 512, ...: at most kGroupVecs), whose
        // group exchange has had this row's partial to complete -- and then
        // moves this row from the stage into the registers and releases the
        // stage.  One stage is held at a time; the others are in flight.
        const bool causal = (a.flags & BSM_FLAG_CAUSAL) != 0;
        unsigned char *y = static_cast<unsigned char *>(a.y);
        const Bounds bdy{nullptr, nullptr, y, y + a.total_elems * E::kSize, a.status};
        const int tid = warp * 32 + lane;
        uint32_t xt = 0;            // group rows this CTA took part in (the exchange sequence)
        uint4 rr[kGroupVecs];       // the row one behind: published, not yet written
        StageMeta rm{};
        uint32_t rx = 0;
        bool rh = false;
        // the row held in rr: poll its K partials (each two words carrying the
        // row's tag) until all are in, combine them in rank order, write this
        // member's part
        auto finish = [&](unsigned long long pre0, unsigned long long pre1) -> bool {
            const uint32_t slot = rx & (kGroupSlots - 1);
            const uint32_t tag = rx + 1;
            const unsigned long long *xs = &xch[2 * static_cast<size_t>(slot) * K];
            float mv[kMaxGroup / 32], sv[kMaxGroup / 32];
            bool in = false;
            const uint64_t t0 = global_timer_ns();
            for (uint32_t tries = 0; tries < (1u << 24); ++tries) {
                bool all = true;
#pragma unroll
                for (int j = 0; j < kMaxGroup / 32; ++j) {
                    const int r2 = lane + 32 * j;
                    mv[j] = -INFINITY;
                    sv[j] = 0.0f;
                    if (r2 < K) {
                        // the first round of rank `lane` was loaded early
                        const bool early = tries == 0 && j == 0;
                        const unsigned long long w0 = early ? pre0 : ld_relaxed_u64(&xs[2 * r2]);
                        const unsigned long long w1 = early ? pre1 : ld_relaxed_u64(&xs[2 * r2 + 1]);
                        all = all && static_cast<uint32_t>(w0 >> 32) == tag && static_cast<uint32_t>(w1 >> 32) == tag;
                        mv[j] = __uint_as_float(static_cast<uint32_t>(w0));
                        sv[j] = __uint_as_float(static_cast<uint32_t>(w1));
                    }
                }
                if (__all_sync(0xFFFFFFFFu, all)) {
                    in = true;
                    break;
                }
                const int give_up = (h.abort_flag || global_timer_ns() - t0 > wait_limit) ? 1 : 0;
                if (__any_sync(0xFFFFFFFFu, give_up))
                    break;
                __nanosleep(32);
            }
            if (!in) {
                if (lane == 0) {
                    atomicOr(a.status, BSM_DEV_TIMEOUT);
                    h.abort_flag = 1;
                }
                return false;
            }
            float M = mv[0];
#pragma unroll
            for (int j = 1; j < kMaxGroup / 32; ++j)
                M = fmaxf(M, mv[j]);
            M = group_max<32>(M);
            float sum = 0.0f;
#pragma unroll
            for (int j = 0; j < kMaxGroup / 32; ++j)
                if (lane + 32 * j < K)
                    sum += mv[j] == M ? sv[j] : sv[j] * ex2((mv[j] - M) * kLog2e);
            sum = group_sum<32>(sum);
            group_write<Tag, Checked>(rr, (rm.C * E::kSize) >> 4, tid, rm.col0, rm.row0, causal, M * kLog2e,
                                      __frcp_rn(sum), y + rm.off * E::kSize, bdy);
            rh = false;
            return true;
        };
        bool failed = false;
        for (uint32_t it = 0;; ++it) {
            const int s = static_cast<int>(it % S);
            const uint32_t ph = (it / S) & 1u;
            // the whole warp gives up together (the shuffles need all lanes)
            if (!__all_sync(0xFFFFFFFFu, mbar_wait_bounded(&h.full[s], ph, &h.abort_flag, wait_limit))) {
                if (lane == 0) {
                    atomicOr(a.status, BSM_DEV_TIMEOUT);
                    h.abort_flag = 1;
                }
                failed = true;
                break;
            }
            const StageMeta mt = h.meta[s];
            if (mt.kind == KIND_DONE)
                break;
            if (mt.kind != KIND_GROUP) {
                __syncwarp();
                if (lane == 0)
                    mbar_arrive(&h.empty[s]);
                continue;
            }
            const int nvec = (mt.C * E::kSize) >> 4;
            const unsigned char *sbuf = stages + static_cast<size_t>(s) * a.stage_bytes;
            Bounds bs = bdy;
            bs.s_lo = sbuf;
            bs.s_hi = sbuf + static_cast<size_t>(mt.C) * E::kSize;
            // the held row's exchange words of rank `lane`, loaded halfway
            // through this row's partial and used after it: late enough that
            // most members have published, early enough that the second half
            // covers the loads' latency
            unsigned long long pre0 = 0, pre1 = 0;
            auto poll = [&]() {
                if (rh && lane < K) {
                    const unsigned long long *xs = &xch[2 * static_cast<size_t>(rx & (kGroupSlots - 1)) * K];
                    pre0 = ld_relaxed_u64(&xs[2 * lane]);
                    pre1 = ld_relaxed_u64(&xs[2 * lane + 1]);
                }
            };
            // this member's (max, sum) of its part, from the stage
            float m_l, s_l;
            group_partial<Tag, Checked>(sbuf, nvec, tid, mt.col0, mt.row0, causal, bs, m_l, s_l, poll);
#pragma unroll
            for (int o2 = 16; o2 >= 1; o2 >>= 1) {
                const float mo2 = __shfl_xor_sync(0xFFFFFFFFu, m_l, o2);
                const float so2 = __shfl_xor_sync(0xFFFFFFFFu, s_l, o2);
                combine_ms(m_l, s_l, mo2, so2);
            }
            // the warps' partials: the last warp to bring its own combines them
            // (a fixed tree over 16 lanes) and publishes the CTA's; nobody
            // waits.  (A warp's partial of row t + 2 comes after its finish of
            // row t, i.e. after row t's publication: two slots by row parity.)
            const int par = xt & 1;
            int last = 0;
            if (lane == 0) {
                h.partial[par][warp] = make_float2(m_l, s_l);
                __threadfence_block();
                last = atomicAdd(&h.xarrive[par], 1u) == static_cast<uint32_t>(kConsumerWarps - 1) ? 1 : 0;
                if (last) {
                    __threadfence_block();
                    h.xarrive[par] = 0u;
                }
            }
            last = __shfl_sync(0xFFFFFFFFu, last, 0);
            if (last) {
                __syncwarp();
                float2 pw = lane < kConsumerWarps ? h.partial[par][lane] : make_float2(-INFINITY, 0.0f);
#pragma unroll
                for (int o2 = kConsumerWarps / 2; o2 >= 1; o2 >>= 1) {
                    const float mo2 = __shfl_xor_sync(0xFFFFFFFFu, pw.x, o2);
                    const float so2 = __shfl_xor_sync(0xFFFFFFFFu, pw.y, o2);
                    combine_ms(pw.x, pw.y, mo2, so2);
                }
                if (lane == 0) {
                    // two self-validating words (value, row tag): 8-byte stores
                    // are single-copy atomic, so a reader that sees the tag
                    // sees the value written with it
                    const uint32_t slot = xt & (kGroupSlots - 1);
                    const unsigned long long tag = static_cast<unsigned long long>(xt + 1) << 32;
                    unsigned long long *w = &xch[2 * (static_cast<size_t>(slot) * K + rank)];
                    st_relaxed_u64(w, tag | __float_as_uint(pw.x));
                    st_relaxed_u64(w + 1, tag | __float_as_uint(pw.y));
                }
            }
            // the previous row: its partials are (nearly) in by now
            if (rh && !finish(pre0, pre1)) {
                failed = true;
                break;
            }
            // this row into the registers; the stage is free
            group_load<Tag, Checked>(rr, sbuf, nvec, tid, bs);
            __syncwarp();
            if (lane == 0)
                mbar_arrive(&h.empty[s]);
            rm = mt;
            rx = xt;
            rh = true;
            ++xt;
        }
        if (!failed && rh)
            finish(0ull, 0ull);
        __syncwarp();
    }
    // the last CTA out resets the queue heads, the claim rings and the
    // exchange counters for the next launch
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        const uint32_t prev = atomicAdd(&a.heads[BSM_MAX_DIES], 1u);
        if (prev == gridDim.x - 1) {
            __threadfence();
            for (int d = 0; d < BSM_MAX_DIES; ++d)
                atomicExch(&a.heads[d], 0u);
            for (int i = 0; i < a.n_groups * kGroupRing; ++i)
                a.ring[i] = 0ull;
            for (int i = 0; i < 2 * a.n_groups * kGroupSlots * a.group_k; ++i)
                a.xch[i] = 0ull;
            __threadfence();
            atomicExch(&a.heads[BSM_MAX_DIES], 0u);
        }
    }
}

}  // namespace

int kernel_set_smem_limit(int bytes)
{
    const void *fns[] = {
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_FORWARD, false>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_FORWARD, false>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_FORWARD, true>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_FORWARD, true>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_BACKWARD, false>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_BACKWARD, false>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_BACKWARD, true>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_BACKWARD, true>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_FORWARD_LONG, false>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_FORWARD_LONG, false>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_FORWARD_LONG, true>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_FORWARD_LONG, true>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_BACKWARD_LONG, false>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_BACKWARD_LONG, false>),
        reinterpret_cast<const void *>(softmax_persistent<F32, OP_BACKWARD_LONG, true>),
        reinterpret_cast<const void *>(softmax_persistent<BF16, OP_BACKWARD_LONG, true>),
        reinterpret_cast<const void *>(softmax_group<F32, false>),
        reinterpret_cast<const void *>(softmax_group<BF16, false>),
        reinterpret_cast<const void *>(softmax_group<F32, true>),
        reinterpret_cast<const void *>(softmax_group<BF16, true>)};
    for (const void *f : fns) {
        cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        if (e != cudaSuccess)
            return static_cast<int>(e);
    }
    return 0;
}

namespace {
template <typename Tag, int Op>
void launch_one(const KernelArgs &a, int grid, size_t smem, cudaStream_t st, bool checked)
{
    // launched with programmatic stream serialisation: the kernel's prologue
    // overlaps the tail of the previous kernel (see griddepcontrol.wait)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
#ifdef BSM_NO_PDL
    cfg.numAttrs = 0;
#endif
    if (checked)
        cudaLaunchKernelEx(&cfg, softmax_persistent<Tag, Op, true>, a);
    else
        cudaLaunchKernelEx(&cfg, softmax_persistent<Tag, Op, false>, a);
}

// Rows over groups of CTAs: a cooperative launch (every CTA resident at once,
// so the members of a group can wait on one another), without the
// programmatic overlap with the previous kernel.
template <typename Tag>
void launch_group(const KernelArgs &a, int grid, size_t smem, cudaStream_t st, bool checked)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(grid));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeCooperative;
    attr[0].val.cooperative = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (checked)
        cudaLaunchKernelEx(&cfg, softmax_group<Tag, true>, a);
    else
        cudaLaunchKernelEx(&cfg, softmax_group<Tag, false>, a);
}
}  // namespace

int launch_softmax(const KernelArgs &a, int dtype, int op, int grid, void *stream, bool checked)
{
    const size_t smem = kSmemHeader + (size_t)a.n_stages * a.stage_bytes;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (op == OP_FORWARD_GROUP) {
        if (dtype == BSM_F32)
            launch_group<F32>(a, grid, smem, st, checked);
        else
            launch_group<BF16>(a, grid, smem, st, checked);
    } else if (op == OP_BACKWARD) {
        if (dtype == BSM_F32)
            launch_one<F32, OP_BACKWARD>(a, grid, smem, st, checked);
        else
            launch_one<BF16, OP_BACKWARD>(a, grid, smem, st, checked);
    } else if (op == OP_BACKWARD_LONG) {
        if (dtype == BSM_F32)
            launch_one<F32, OP_BACKWARD_LONG>(a, grid, smem, st, checked);
        else
            launch_one<BF16, OP_BACKWARD_LONG>(a, grid, smem, st, checked);
    } else if (op == OP_FORWARD_LONG) {
        if (dtype == BSM_F32)
            launch_one<F32, OP_FORWARD_LONG>(a, grid, smem, st, checked);
        else
            launch_one<BF16, OP_FORWARD_LONG>(a, grid, smem, st, checked);
    } else {
        if (dtype == BSM_F32)
            launch_one<F32, OP_FORWARD>(a, grid, smem, st, checked);
        else
            launch_one<BF16, OP_FORWARD>(a, grid, smem, st, checked);
    }
    return static_cast<int>(cudaGetLastError());
}

}  // namespace bsm
