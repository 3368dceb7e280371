// bsm_internal.h -- types shared by the kernels (.cu) and the host side
// (.cpp) of libbsm.  Not part of the public ABI.
#pragma once

#include <cstdint>

#include "../../include/bsm.h"

namespace bsm {

// One patch ("batch or patch", Sec. 4: the unit of work the scheduler places):
// nrows consecutive rows of C elements, contiguous in x and y from element
// `off`.  Under the RR and WHOLE_GPU policies a patch stays inside one slice;
// under the queue policies it may run on into following slices of the same
// shape (R x C, packed back to back).  The first row is row `row0` of its
// slice and every slice of the patch has R rows, so row r of the patch is row
// (row0 + r) mod R of its slice (the causal mask needs it).
struct Item {
    int64_t off;
    int32_t C;
    int32_t nrows;
    int32_t row0;
    int32_t R;
};
static_assert(sizeof(Item) == 24, "Item layout");

// How a CTA finds its next patch.
enum PullMode : int32_t {
    PULL_STATIC = 0,    // CTA b takes items item_begin + b, + b + G, ... (< item_end)
    PULL_RR_SLICE = 1,  // CTA b takes every patch of slices b, b + G, ... (Sec. 3 RR)
    PULL_QUEUE = 2      // CTA pulls from its die's queue, then (steal) the others'
};

// Patches fetched per producer round trip.
constexpr int kFetch = 4;

constexpr int kMaxStages = 8;
constexpr int kConsumerWarps = 16;
constexpr int kThreads = (kConsumerWarps + 1) * 32;  // + one producer warp
constexpr int kSmemHeader = 1024;                     // barriers + stage metadata
// Smallest stage (three fit the shared memory).  Each stage has a fixed cost
// (wait, metadata, dispatch, release) that larger stages amortise; measured
// over 32 KiB stages: bf16 +11 % causal 512-wide rows, +16 % 32 x 128 slices;
// fp32 +2 % 512 x 512 slices (+4 % with die queues), backward +2 %; 72 KiB
// and more (two or three stages) is slower again.
constexpr int kMinStageBytes = 64 * 1024;

// What the kernel computes on every row.
enum Op : int32_t {
    OP_FORWARD = 0,     // y = softmax(x [+ causal mask])
    OP_BACKWARD = 1,    // y = x * (x2 - rowsum(x * x2)): x = softmax output, x2 = its gradient
    OP_FORWARD_LONG = 2, // OP_FORWARD for plans with rows longer than a stage (two passes)
    OP_BACKWARD_LONG = 3, // OP_BACKWARD for plans with rows longer than half a stage (two passes)
    OP_FORWARD_GROUP = 4 // OP_FORWARD of rows split over groups of CTAs (one read; see KernelArgs)
};

// Rows split over groups of CTAs (OP_FORWARD_GROUP): group g is CTAs
// [g*K, g*K + K); its rank-0 CTA claims rows and announces them in the
// group's ring of kGroupRing claim words (row sequence number + 1 in the high
// half, the row's position in the table in the low half); each member stages
// its part of the row and publishes its (max, sum) in one of kGroupSlots
// exchange slots as two words (the row sequence number + 1 in the high half
// of each, max or sum in the low half).  Rings and exchange words are reset
// by the last CTA of every launch.
constexpr int kGroupRing = 16;
constexpr int kGroupSlots = 4;
constexpr int kMaxGroup = 128;
// A member's part is held in registers while its group exchanges partials:
// at most kGroupVecs 16-byte vectors per consumer thread, i.e. parts of at
// most kGroupVecs * 16 * 512 bytes = 64 KiB.
constexpr int kGroupVecs = 8;

// A row longer than one stage is cut into segments of whole stage-sized
// chunks, each its own patch (nrows = 1, off/C = the segment).  An execute
// then takes two launches: in phase 0 every segment streams its chunks and
// leaves a partial in partials[2*part] -- (max, sum of exp(v - max)) forward,
// (<y, dy>, 0) backward -- while short rows are finished; in phase 1 every
// segment combines its row's partials [part_first, part_first + part_count)
// in that order (the same for every segment and every policy) and streams
// its chunks again to write the output.  part_count = 0: a short-row patch.
struct LongSeg {
    int32_t col0;               // column of the segment's first element in its row
    int32_t part;
    int32_t part_first;
    int32_t part_count;
};

struct KernelArgs {
    const void *x;
    const void *x2;             // OP_BACKWARD: the upstream gradient
    void *y;
    int64_t total_elems;        // extent of x and y, elements (bounds checks)
    const Item *items;
    int32_t n_items;
    int32_t mode;               // PullMode
    int32_t item_begin, item_end;           // PULL_STATIC
    const int32_t *slice_first_item;        // PULL_RR_SLICE: n_slices + 1 entries
    int32_t n_slices;
    int32_t n_queues;                       // PULL_QUEUE: items are stored in queue
    int32_t queue_begin[BSM_MAX_DIES];      // order; queue d is items[begin, begin+len)
    int32_t queue_len[BSM_MAX_DIES];
    int32_t steal;
    uint32_t *heads;            // BSM_MAX_DIES queue heads + 1 exit counter; self-resetting
    const int8_t *sm_die;       // die of each %smid (NULL: all die 0)
    int32_t stage_bytes;
    int32_t n_stages;
    uint32_t flags;
    uint32_t *status;           // sticky device status word
    uint64_t wait_limit_ns;     // bound of every pipeline wait (0 = the 2 s default)
    uint32_t debug;             // fault injection for tests: KDEBUG_* bits
    // rows longer than a stage (OP_*_LONG): see LongSeg
    const LongSeg *segs;        // per patch, in the order of `items`; NULL: no long rows
    float *partials;            // 2 floats per segment
    int32_t phase;              // 0: segments leave their partials; 1: combine and write
    // rows split over groups of CTAs (OP_FORWARD_GROUP): items are whole rows
    int32_t group_k;            // CTAs per group (2..kMaxGroup); the grid is n_groups * group_k
    int32_t n_groups;
    unsigned long long *ring;   // n_groups x kGroupRing claim words
    unsigned long long *xch;    // n_groups x kGroupSlots x group_k x 2 tagged words: max, sum
};

// Test-only fault injection (bsm_plan_debug).
constexpr uint32_t KDEBUG_WITHHOLD_STAGE0 = 1u;   // producer never fills stage 0 of its first round

// One output tile of the batched matrix product: rows [m0, m0 + 128) and
// columns [n0, n0 + BN) of slice `slice`.
struct GemmItem {
    int32_t slice, m0, n0, pad;
};

struct GemmArgs {
    void *c;                    // B x M x N output (bf16 or fp32)
    int32_t B, M, N, K;
    const GemmItem *items;
    int32_t n_items;
    int32_t mode;               // PullMode
    int32_t item_begin, item_end;
    const int32_t *slice_first_item;
    int32_t n_slices;
    int32_t n_queues;
    int32_t queue_begin[BSM_MAX_DIES];
    int32_t queue_len[BSM_MAX_DIES];
    int32_t steal;
    uint32_t *heads;
    const int8_t *sm_die;
    int32_t n_stages;
    int32_t epi_bufs;               // 2..4 store buffers per epilogue warp
    int32_t kbs;                    // K blocks of 64 per stage (1, 2 or 4)
    int32_t identity;               // items in natural order: computed, not read
    int32_t tiles_m, tiles_n;       // row / column blocks per slice
    uint32_t *status;
};

// Batched matrix product kernel (bsm_bmm.cu).  tmap_a / tmap_b / tmap_c point
// at host CUtensorMap objects (C: boxes of 32 rows x 128 bytes, 128-byte
// swizzle).  Return cudaError_t values.
int launch_bmm(const void *tmap_a, const void *tmap_b, const void *tmap_c, const GemmArgs &a, int bn,
               bool out_bf16, int grid, void *stream);
int gemm_set_smem_limit(int bytes);
int gemm_stage_bytes(int bn);
// shared memory of one launch besides the stages (header, slack, epilogue
// store buffers: epi_bufs of 4 KiB per epilogue warp with work)
int gemm_fixed_smem(int bn, bool out_bf16, int epi_bufs);

// Launch the persistent softmax kernel (bsm_kernels.cu).  Returns a
// cudaError_t value (0 = success).
int launch_softmax(const KernelArgs &a, int dtype, int op, int grid, void *stream, bool checked);
// Raise the dynamic shared-memory limit of both kernel instances.
int kernel_set_smem_limit(int bytes);

// Probe kernels (bsm_probe.cu).  All synchronous; return cudaError_t values.
int probe_latency_run(const void *buf, const int64_t *line_off_dev, int n_lines, int reps,
                      int grid, float *lat_dev, uint32_t *claim_dev);
int probe_map_run(const void *buf, int64_t bytes, int64_t chunk, int reps, const int8_t *sm_die_dev, int want_die,
                  int n_sm, uint32_t *counter_dev, float *lat_dev);
// Die-map check (bsm_probe.cu): SMs of die d read the chunks listed for d.
int die_check_run(const void *buf, int64_t n_chunks, int64_t chunk, const int32_t *list0, int64_t len0,
                  const int32_t *list1, int64_t len1, uint32_t *ctr, const int8_t *sm_die_dev, int n_sm,
                  uint32_t *sink, float *ms);

// Die of every chunk of a device buffer (bsm_topology.cpp): timed from an SM
// of each of the probe's dies, or of each group of sm_group when given.
int addr_die_map_host(int device, const void *ptr, int64_t bytes, int64_t chunk, int8_t *die_out,
                      const int8_t *sm_group = nullptr);

// Remember a failing CUDA call for bsm_last_cuda_error (bsm_api.cpp);
// returns BSM_ERR_CUDA.
int record_cuda_error(int cuda_error, const char *where);

// Sticky status bits left by bsm_softmax_noalloc on `device` (bsm_noalloc.cu;
// 0 if it never ran there); clear != 0 zeroes them afterwards.
int noalloc_status(int device, uint32_t *bits, int clear);
// Fault injection for bsm_softmax_noalloc's launches (bsm_plan_debug with a
// null plan): BSM_DEBUG_NONE or BSM_DEBUG_WITHHOLD_STAGE.
int noalloc_debug(int what, int64_t arg);

// Host planner (bsm_planner.cpp).
int schedule_host(const bsm_schedule_desc *d, bsm_schedule_out *out);

}  // namespace bsm
