/*
 * bsm.h -- C ABI of libbsm: batched row-wise softmax over many slices, with
 * the slices scheduled onto the GPU's SMs by a selectable policy.
 *
 * What is computed (Sec. 2 of "An optimal scheduling architecture for
 * accelerating batch algorithms on Neural Network processor architectures",
 * Nyshadham et al.: SOFTMAX on every 512 x 512 slice of a (512*384) x 512
 * tensor; Sec. 6, SOFTMAX table).  For slice s with R_s rows and C_s columns
 * stored row-major at element offset off_s, and every row r of it:
 *     v[c] = x[r,c] + M[r,c]   (M = 0; with BSM_FLAG_CAUSAL, M = -inf for c > r)
 *     y[r,c] = exp(v[c] - max v) / sum_c' exp(v[c'] - max v)
 * A row holding NaN or +inf, or a row that is entirely -inf, comes out NaN
 * (the formula gives 0/0 or inf - inf there).
 *
 * How slices are scheduled (the policies) -- Sec. 3 and Sec. 4:
 *   BSM_POLICY_WHOLE_GPU  Sec. 3, first previous solution: one slice after
 *                         another, each spread over the whole device (one
 *                         launch per slice).
 *   BSM_POLICY_RR         Sec. 3, second previous solution: slice i runs on
 *                         compute unit (i mod G), statically.
 *   BSM_POLICY_CBMF       Sec. 4.1, Cluster Beamforming: every patch (a block
 *                         of rows of one slice) goes to the die whose memory
 *                         holds most of its bytes (ties: seeded fair coin);
 *                         the SMs of that die take the die's patches in order.
 *   BSM_POLICY_CBMF_LB    Sec. 4.1 + Sec. 4.2: CBMF followed by the weighted
 *                         load balance (patches moved from the over-loaded die
 *                         to the other, weighted by inverse latency), plus
 *                         run-time stealing once a die's own queue is empty.
 *   BSM_POLICY_DYNAMIC    Not in the paper: one device-wide queue of patches,
 *                         every SM pulls the next one (the locality-blind
 *                         dynamic schedule CBMF is measured against).
 *   BSM_POLICY_MINIMAX    Sec. 4.2, general form: patches assigned to dies to
 *                         minimise the largest per-SM finish time, a patch's
 *                         cost depending on its distance to the die (near /
 *                         far latency); solved by longest-patch-first, the
 *                         queues then run longest first, with stealing.
 * Every policy computes every row with the same device routine, chosen only
 * by the row length, so y is bit-identical across policies.
 *
 * Conventions shared by every entry point below:
 *   - x and y are device pointers owned by the caller.  They must stay valid
 *     until the work queued on `stream` completes.  Host arrays passed in are
 *     copied; the caller keeps ownership.
 *   - Calls return a bsm_status; no C++ exception crosses the ABI.  Argument
 *     checks are synchronous.  The launches are asynchronous on `stream`
 *     (NULL = the legacy default stream); a fault detected inside a kernel is
 *     recorded in a sticky per-device status word (bsm_device_status).
 *   - Alignment: x and y 16-byte aligned, every slice's byte offset and every
 *     row's byte length (C * element size) a multiple of 16; otherwise
 *     BSM_ERR_MISALIGNED.
 *   - In place (x == y) is allowed; partially overlapping x and y are not
 *     (BSM_ERR_INVALID_ARG).
 *   - Row length: a row of up to bsm_max_row_bytes() (half of it for the
 *     backward pass, where y and dy share a stage) is read once from one
 *     shared-memory stage.  Longer rows go through the stages in chunks, in
 *     two passes -- a running maximum and rescaled sum (backward: the dot
 *     product), then the output.  A row of two chunks whose halves fit three
 *     stages (with the batch's shorter rows) stays staged between the passes
 *     and is read once; longer rows are read again, all but their last
 *     chunk.  When a batch has fewer such rows than two per SM, each is cut
 *     into segments spread over the SMs and the execute takes two launches
 *     (segment partials, then combine and write); otherwise each row stays
 *     on one SM within one launch.  Forward rows of 5 to 32 parts of at most
 *     64 KiB, enough of them to fill two thirds of the groups'
 *     waves, are instead split over groups of K CTAs (K = ceil(row / 64
 *     KiB); n_sm / K groups) in one cooperative launch: each CTA stages one
 *     part, the group exchanges (max, sum) partials through global memory
 *     and every element is read once.  Which path a row takes depends on the
 *     rows of the batch and the device, never on the policy: every policy
 *     gives the same bits.
 */
#ifndef BSM_H
#define BSM_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* A cudaStream_t.  NULL selects the legacy default stream. */
typedef struct CUstream_st *bsm_stream_t;

typedef enum {
    BSM_OK = 0,
    BSM_ERR_INVALID_ARG = 1,   /* null / negative / inconsistent arguments */
    BSM_ERR_MISALIGNED = 2,    /* 16-byte alignment rule broken */
    BSM_ERR_UNSUPPORTED = 3,   /* shape outside a kernel's limits, too many patches */
    BSM_ERR_CUDA = 4,          /* a CUDA runtime call failed */
    BSM_ERR_DEVICE_BOUNDS = 5, /* a kernel met a patch outside the buffers */
    BSM_ERR_TIMEOUT = 6,       /* a kernel wait gave up after its time limit */
    BSM_ERR_NO_DEVICE = 7,     /* no usable CUDA device */
    BSM_ERR_NOMEM = 8,         /* host or device allocation failed */
    BSM_ERR_TOO_LARGE = 9      /* more patches than bsm_softmax_noalloc's fixed scratch holds */
} bsm_status;

typedef enum { BSM_F32 = 0, BSM_BF16 = 1 } bsm_dtype;   /* input type == output type */

typedef enum {
    BSM_POLICY_WHOLE_GPU = 0,
    BSM_POLICY_RR = 1,
    BSM_POLICY_CBMF = 2,
    BSM_POLICY_CBMF_LB = 3,
    BSM_POLICY_DYNAMIC = 4,
    BSM_POLICY_MINIMAX = 5
} bsm_policy;

#define BSM_FLAG_CAUSAL 1u     /* additive -inf mask above each slice's diagonal */

#define BSM_MAX_DIES 4
#define BSM_MAX_SM 256

/* Device-side status bits (bsm_device_status). */
#define BSM_DEV_BOUNDS 1u      /* a patch fell outside the buffers or a stage; skipped */
#define BSM_DEV_TIMEOUT 2u     /* a pipeline wait ran out of time; the CTA gave up */
#define BSM_DEV_CHECK 4u       /* the checking kernel caught an out-of-range access; skipped */

/*
 * Softmax over B slices of R x C stored back to back, i.e. a (B*R) x C
 * row-major tensor (the layout of Sec. 2).  Equivalent to bsm_softmax_ex with
 * flags = 0.  The plan (patch table, die queues) is built on first use for a
 * given (device, x, y, shape, dtype, policy, flags) and cached.  Calls that
 * share a cached plan share its queue counters, which the last CTA of an
 * execution resets.  Such calls must therefore not run at the same time on
 * different streams; they write the same y anyway, so order them.
 *   x, y    device pointers, B*R*C elements of `dtype` each.
 *   B, R, C B >= 0, R >= 0, C >= 1; B*R*C < 2^62.
 *   dtype   bsm_dtype; policy bsm_policy.
 * Errors: BSM_ERR_INVALID_ARG, BSM_ERR_MISALIGNED, BSM_ERR_UNSUPPORTED,
 * BSM_ERR_CUDA, BSM_ERR_NOMEM.  B*R == 0 returns BSM_OK and launches nothing.
 */
int bsm_softmax(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype,
                int policy, bsm_stream_t stream);

/* bsm_softmax with flags (BSM_FLAG_CAUSAL: M[r,c] = -inf for c > r, r the row
 * inside its slice). */
int bsm_softmax_ex(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype,
                   int policy, uint32_t flags, bsm_stream_t stream);

/*
 * bsm_softmax_ex on HOST buffers.  Page-locked (pinned, e.g. cudaHostAlloc or
 * cudaHostRegister) buffers are read and written by the kernel directly over
 * the CPU-GPU link (NVLink-C2C on Grace-Blackwell): no device memory, both
 * link directions in use at once.  Pageable buffers go through a staged
 * pipeline: the batch is cut into chunks of whole slices (about 48 MiB of
 * input each); each chunk is copied to a device staging buffer, processed and
 * copied back, on three streams of the library with two staging buffers, so
 * that copying in, computing and copying out of consecutive chunks overlap;
 * the staging buffers (2 x 2 x chunk bytes) are allocated on first use and
 * kept per device, and such calls on one device are serialised on the host.
 * Asynchronous with respect to `stream`: the work starts after what is
 * already queued on `stream`, and `stream` waits for its end; synchronise
 * `stream` before reading y_host.
 *   x_host, y_host  host pointers, B*R*C elements each; may be equal.
 *   B, R, C, dtype, policy, flags  as bsm_softmax_ex.
 * Errors: as bsm_softmax_ex.
 */
int bsm_softmax_host(const void *x_host, void *y_host, int64_t B, int64_t R, int64_t C, int dtype,
                     int policy, uint32_t flags, bsm_stream_t stream);

/*
 * Ragged batch: slice s has rows[s] x cols[s] elements at element offset
 * offsets[s] of x (and of y).  The paper's slices are uniform (Sec. 2); its
 * load balance (Sec. 4.2) exists because patches differ in size, and a batch
 * of slices of different shapes is where they do.  The paper has no call of
 * this shape; it is the ragged form the scheduling contract asks for, with
 * the same per-row computation as bsm_softmax.  offsets/rows/cols are HOST arrays of
 * num_slices entries, copied.  Slices must not overlap each other; they need
 * not be contiguous or ordered.  Same errors as bsm_softmax.
 */
int bsm_softmax_ragged(const void *x, void *y, int64_t num_slices, const int64_t *offsets,
                       const int32_t *rows, const int32_t *cols, int dtype, int policy,
                       uint32_t flags, bsm_stream_t stream);

/*
 * bsm_softmax_ex without any allocation -- for callers that cannot allocate
 * device memory: code living inside a pre-reserved memory pool or arena (a
 * server that sized the whole device up front, a framework whose allocator
 * must account for every byte), or a latency-critical path that must not
 * pick up the device-wide synchronisation of cudaMalloc/cudaFree.  The paper
 * has no counterpart; this is a deployment variant of the dynamic schedule.
 *
 * The same kernel, row routine and patches as bsm_softmax_ex with
 * BSM_POLICY_DYNAMIC, for B slices of R x C packed back to back, so the
 * results are bit for bit the same -- for rows that fit one shared-memory
 * stage: at most BSM_NOALLOC_MAX_ROW_BYTES (C * element size), and at most
 * the device's own stage limit (half its opt-in shared memory per block less
 * 1 KiB, rounded down to 128 bytes: the same 113 KiB on GB300).  Longer rows
 * get BSM_ERR_UNSUPPORTED here (bsm_softmax_ex streams them in two passes,
 * which needs buffers this entry point does not have).
 *
 * Instead of a plan, the patch table and queue counters live in one fixed
 * device array inside the library: every GPU that loads the library holds it
 * (about 1.5 MiB) until the process exits.  The first call on a device, with
 * that device current, looks the array's address up (cudaGetSymbolAddress):
 * make that first call before any stream capture.  Every call shares the
 * array and it keeps the last call's contents; each call rewrites the patch
 * table and zeroes the counters on `stream` first, so calls that overlap on
 * the GPU (other streams, unordered threads) race.  Device-side error bits
 * of this entry point are sticky in the array: bsm_device_status reports
 * them (OR-ed with the library's own word) and bsm_device_status_clear
 * zeroes them.  Nothing is allocated and nothing synchronises.
 *   x, y, B, R, C, dtype, flags, stream: as bsm_softmax_ex.
 * Errors: as bsm_softmax_ex; BSM_ERR_UNSUPPORTED for a row past the limit
 * above; BSM_ERR_TOO_LARGE when the batch needs more than
 * BSM_NOALLOC_MAX_PATCHES patches (a patch is the rows that fill one 64 KiB
 * shared-memory stage: for 2 KiB rows, 32 rows; 65536 patches cover 4 GiB of
 * input).  The row and patch limits are checked before the device is touched.
 */
#define BSM_NOALLOC_MAX_PATCHES 65536
#define BSM_NOALLOC_MAX_ROW_BYTES 115712   /* 113 KiB */
int bsm_softmax_noalloc(const void *x, void *y, int64_t B, int64_t R, int64_t C, int dtype,
                        uint32_t flags, bsm_stream_t stream);

/*
 * Backward pass of the batched softmax (Sec. 1: the batch algorithms run in
 * the forward or the backward pass) over the same slices and the same
 * scheduler: for every row, given the forward output y and the upstream
 * gradient dy,
 *     dx[c] = y[c] * (dy[c] - sum_c' y[c'] * dy[c'])
 * (the vector-Jacobian product of the row softmax; with a causal forward the
 * masked y are 0 and so are their dx).  y, dy, dx: device pointers, B*R*C
 * elements of `dtype`; dx may equal y or dy; other overlaps are rejected.
 * Rows of any length (see "Row length" above).
 * Same scheduling policies, errors and alignment rules as bsm_softmax.
 */
int bsm_softmax_backward(const void *y, const void *dy, void *dx, int64_t B, int64_t R, int64_t C,
                         int dtype, int policy, bsm_stream_t stream);

/* Ragged form of bsm_softmax_backward (slices as in bsm_softmax_ragged). */
int bsm_softmax_backward_ragged(const void *y, const void *dy, void *dx, int64_t num_slices,
                                const int64_t *offsets, const int32_t *rows, const int32_t *cols,
                                int dtype, int policy, bsm_stream_t stream);

/*
 * Batched matrix product, the paper's other batch algorithm (Sec. 6: batch
 * 384 of (512 x 64) x (64 x 512) and of (512 x 512) x (512 x 64)), on the
 * tensor cores, with the output tiles (128 x 64/128/256 of one slice) as the
 * patches of the same scheduling policies:
 *     C_s[m, n] = sum_k A_s[m, k] * Bt_s[n, k]        (C_s = A_s Bt_s^T)
 *   a   device, B x M x K bf16, row-major (slice s at s*M*K)
 *   bt  device, B x N x K bf16, row-major: the second factor TRANSPOSED, i.e.
 *       with the reduction dimension contiguous (attention's K matrix as it
 *       is; for P*V pass V^T)
 *   c   device, B x M x N, out_dtype BSM_F32 or BSM_BF16 (fp32 accumulation,
 *       rounded to nearest even for bf16)
 *   M a multiple of 128, N of 64, K of 64 (else BSM_ERR_UNSUPPORTED);
 *   pointers 16-byte aligned; c must not overlap a or bt.
 * Plans are cached like bsm_softmax's, with the same rule: calls that share
 * one (same pointers, shapes, dtype, policy) must not run at the same time on
 * different streams.  Errors as bsm_softmax.
 */
int bsm_bmm(const void *a, const void *bt, void *c, int64_t B, int64_t M, int64_t N, int64_t K,
            int out_dtype, int policy, bsm_stream_t stream);

/*
 * bsm_bmm with the shared-memory split chosen by the caller (0 = automatic,
 * as bsm_bmm): n_stages operand stages in flight per SM (2..8), each holding
 * k_blocks_per_stage (1, 2 or 4; must divide K/64) blocks of 64 columns of
 * K of the 128-row A tile and of the N_tile-row Bt tile, fetched with one
 * copy per operand; epi_bufs 4 KiB output store buffers per epilogue warp
 * (2..4).  A split that does not fit in one SM's shared memory, or a block
 * count that does not divide K/64, returns BSM_ERR_UNSUPPORTED; out-of-range
 * values BSM_ERR_INVALID_ARG.  Results do not depend on the split.
 */
int bsm_bmm_ex(const void *a, const void *bt, void *c, int64_t B, int64_t M, int64_t N, int64_t K,
               int out_dtype, int policy, int n_stages, int epi_bufs, int k_blocks_per_stage,
               bsm_stream_t stream);

/* ---- plans: build the schedule once ("upfront", Sec. 5), run it many times ---- */

typedef struct bsm_plan bsm_plan;

typedef struct {
    const void *x;              /* device input */
    void *y;                    /* device output (may equal x) */
    int64_t num_slices;
    const int64_t *offsets;     /* host, element offsets; NULL = packed back to back */
    const int32_t *rows;        /* host, num_slices entries */
    const int32_t *cols;        /* host, num_slices entries */
    int32_t dtype;              /* bsm_dtype */
    int32_t policy;             /* bsm_policy */
    uint32_t flags;             /* BSM_FLAG_* */
    int32_t rows_per_item;      /* rows per patch at most; 0 = as many as fill one stage
                                   (the queue policies cut a batch of fewer such patches
                                   than SMs into ceil(rows / SMs)-row patches: one per SM) */
    uint64_t tie_seed;          /* seed of the CBMF equal-share coin */
    int32_t lb_weighted;        /* CBMF_LB: 1 = weights from measured latency, 0 = equal */
    int32_t count_output_bytes; /* CBMF: 1 = a patch's bytes on a die count x and y */
    int32_t device;             /* -1 = the current device */
    int32_t op;                 /* BSM_OP_FORWARD (default) or BSM_OP_BACKWARD */
    const void *x2;             /* BSM_OP_BACKWARD: the upstream gradient dy (x holds y) */
} bsm_plan_desc;

#define BSM_OP_FORWARD 0        /* y = softmax(x) */
#define BSM_OP_BACKWARD 1       /* y = x * (x2 - rowsum(x * x2)): dx from y = x and dy = x2 */

/* Fill a descriptor with the defaults (rows_per_item 0, tie_seed 0x2002070600,
 * lb_weighted 1, count_output_bytes 1, device -1, offsets NULL). */
int bsm_plan_desc_init(bsm_plan_desc *d);

/* Build a plan: validate, cut slices into patches, and for CBMF / CBMF_LB
 * probe the topology (cached per device) and the die of every chunk of x and
 * y, then run the Sec. 4.1 / 4.2 steps on the host and upload the tables.
 * A WHOLE_GPU plan of up to 4096 launches also captures them as one CUDA
 * graph (executed without per-kernel launches; a debug setting or the
 * self-checking kernels bring back kernel-by-kernel launches).
 * Synchronous; allocates device memory owned by the plan. */
int bsm_plan_create(bsm_plan **plan, const bsm_plan_desc *d);

/* Launch the plan on `stream` (async): the persistent kernel walks the
 * table built up front (Sec. 5: the scheduler fills its mapping table once,
 * then feeds patch coordinates to one templated kernel; Sec. 4.1: each
 * compute unit takes its bank's patches in order).  Allocates nothing and
 * does not synchronise.  Executions of one plan must not overlap in time (they share
 * the plan's queue counters and its long-row partials): keep them on one
 * stream, or order them. */
int bsm_plan_execute(const bsm_plan *plan, bsm_stream_t stream);

typedef struct {
    int32_t policy;
    int32_t n_die;              /* dies the schedule used (1 if not separable) */
    int64_t n_items;            /* patches */
    int64_t N[BSM_MAX_DIES];    /* Sec. 4.1: patches with any byte on die d */
    int64_t L[BSM_MAX_DIES];    /* Sec. 4.1: patches assigned to die d */
    int64_t overlap_items;      /* patches on more than one die */
    int64_t tie_items;          /* patches resolved by the coin */
    int64_t moved_items;        /* Sec. 4.2: patches moved by the load balance */
    int64_t queue_items[BSM_MAX_DIES];
    int64_t queue_bytes[BSM_MAX_DIES];
    double est_finish_before[BSM_MAX_DIES];  /* per-die estimated finish, LB input */
    double est_finish_after[BSM_MAX_DIES];   /* same after LB */
    int32_t stage_bytes;        /* shared-memory stage size */
    int32_t n_stages;           /* stages per CTA */
    int32_t grid;               /* CTAs per launch */
    int32_t launches;           /* launches per execute (WHOLE_GPU: one per slice) */
    int32_t steal;              /* 1 if CTAs steal from other dies' queues */
    int64_t map_chunk_bytes;    /* granularity of the address->die map used */
    double plan_ms;             /* host time spent in bsm_plan_create */
    int64_t long_items;         /* rows longer than a stage (group rows included) */
    int64_t group_rows;         /* rows split over groups of CTAs (one cooperative launch) */
    int32_t group_k;            /* CTAs per group */
    int32_t n_groups;           /* groups of that launch */
} bsm_plan_stats;

int bsm_plan_get_stats(const bsm_plan *plan, bsm_plan_stats *out);
void bsm_plan_destroy(bsm_plan *plan);

/* ---- the schedule a plan was built with (for checking it against an
 * independent restatement of Sec. 4.1 / 4.2, and for diagnosis) ----
 * bsm_plan_get_schedule fills the scalar fields always; each array pointer
 * the caller sets (non-NULL) receives its data -- a first call with all
 * arrays NULL gives the sizes.  Host only; no device access.
 *   queue    n_items entries: for every queue slot, the index of its patch in
 *            slice order (the order of bsm_plan_layout_host's phase 0); the
 *            slots of die d's queue are [queue_begin[d], + queue_len[d]).
 *            Written only for the queue policies (n_queues > 0).
 *   x_map    n_map_chunks entries: die of every map_chunk_bytes chunk of x,
 *            as probed at plan creation (CBMF, CBMF_LB, MINIMAX on a
 *            separable device; otherwise n_map_chunks = 0).
 *   y_map    the same for y, when the table counted output bytes and y != x.
 *   moved    n_moved entries: the patches the Sec. 4.2 balance moved, in
 *            order (CBMF_LB).
 * units, l_near, l_far and tie_seed are the planner's other inputs (SMs per
 * die, integer latency weights, the tie coin's seed).  Returns
 * BSM_ERR_INVALID_ARG for a null plan or out. */
typedef struct {
    int32_t n_queues;           /* 0: the policy takes patches statically (RR, WHOLE_GPU) */
    int32_t count_output_bytes;
    int32_t queue_begin[BSM_MAX_DIES];
    int32_t queue_len[BSM_MAX_DIES];
    int32_t units[BSM_MAX_DIES];
    int64_t l_near, l_far;
    uint64_t tie_seed;
    int64_t n_items;
    int64_t map_chunk_bytes;
    int64_t n_map_chunks;
    int64_t n_moved;
    int32_t *queue;
    int8_t *x_map;
    int8_t *y_map;
    int32_t *moved;
} bsm_plan_schedule;

int bsm_plan_get_schedule(const bsm_plan *plan, bsm_plan_schedule *out);


/* ---- the patch table alone, on the host (no GPU needed) ----
 * Cuts the descriptor's slices into patches exactly as bsm_plan_create does,
 * for a device with n_sm SMs and smem_optin bytes of opt-in shared memory per
 * block (Sec. 4: a patch is a block of consecutive rows of one slice -- under
 * the queue policies, of back-to-back slices of one shape -- that fills at
 * most one stage; a row longer than a stage is one patch, or, when such rows
 * are too few to fill the SMs twice, several segments of whole chunks that
 * run in two launches).  d->x, d->y and d->x2 only take part in the
 * alignment and overlap checks and are never dereferenced.  Phase-0 patches
 * come in slice order (before any queue ordering), phase-1 segments in the
 * order the second launch takes them.  At most cap0 / cap1 records are
 * written to phase0 / phase1 (host memory owned by the caller; NULL with a
 * capacity of 0); *out always receives the counts, so a first call with both
 * capacities 0 sizes the arrays.  Returns BSM_ERR_INVALID_ARG for a null d or
 * out, n_sm outside 1..BSM_MAX_SM, smem_optin outside (1024, 1 MiB] or a
 * capacity without an array, and the errors of bsm_plan_create's validation
 * (BSM_ERR_MISALIGNED, BSM_ERR_UNSUPPORTED when fewer than two stages fit). */
typedef struct {
    int64_t elem_offset;        /* first element of the patch in x and y */
    int32_t cols;               /* elements of each of its rows (a segment: its length) */
    int32_t nrows;              /* rows in the patch (1 for a long row) */
    int32_t row0;               /* index of its first row within its slice */
    int32_t slice_rows;         /* R of that slice */
    int32_t col0;               /* long rows: the segment's first column; else 0 */
    int32_t part_count;         /* long rows: segments of the row (1 = the whole row); else 0 */
} bsm_patch;

typedef struct {
    int64_t stage_bytes;        /* bytes per shared-memory stage */
    int32_t n_stages;           /* stages per CTA */
    int32_t group_k;            /* CTAs per group of the rows split over groups (0: none) */
    int64_t n_patches;          /* phase 0 (the first or only launch), group rows included */
    int64_t n_patches_phase1;   /* segments of rows cut into several (the second launch) */
    int64_t long_rows;          /* rows longer than a stage */
} bsm_layout;

int bsm_plan_layout_host(const bsm_plan_desc *d, int32_t n_sm, int64_t smem_optin, bsm_patch *phase0,
                         int64_t cap0, bsm_patch *phase1, int64_t cap1, bsm_layout *out);

/* The patch records as the kernel reads them from the plan's device table
 * (queue policies: in queue order, so that slot k holds patch queue[k]),
 * phase 0 or 1 (the second launch of rows cut into segments).  At most cap
 * records go to out (host, caller-owned); *n_out receives the count.
 * Synchronous (a device-to-host copy).  BSM_ERR_INVALID_ARG for a null plan
 * or n_out, a phase other than 0/1, or a capacity without an array. */
int bsm_plan_device_table(const bsm_plan *plan, int phase, bsm_patch *out, int64_t cap,
                          int64_t *n_out);

/* Fault injection on one plan, for the library's failure-detection tests
 * (nothing here faults, traps or hangs the GPU).  plan = NULL applies
 * BSM_DEBUG_WITHHOLD_STAGE / BSM_DEBUG_NONE to the bsm_softmax_noalloc
 * launches that follow, in every thread (its timeout then shows in
 * bsm_device_status); BSM_DEBUG_CORRUPT_PATCH needs a plan.
 *   BSM_DEBUG_WITHHOLD_STAGE  later executes never fill the first shared-memory
 *                             stage of each CTA, so the consumers' bounded waits
 *                             run out; arg = the wait limit in ns (> 0).  The
 *                             kernel sets BSM_DEV_TIMEOUT and every CTA exits.
 *   BSM_DEBUG_CORRUPT_PATCH   the device patch table entry at position arg is
 *                             rewritten to start past the end of the buffers; the
 *                             kernel's bounds check skips it and sets
 *                             BSM_DEV_BOUNDS (its rows are not written).  Positions
 *                             past the regular table's address the table of rows
 *                             split over groups of CTAs (every member of the
 *                             group skips such a row alike).
 *   BSM_DEBUG_NONE            restore the normal wait limit and switch the
 *                             withheld stage off (a corrupted entry stays).
 * Synchronous.  Returns BSM_ERR_INVALID_ARG for an unknown `what` or arg. */
#define BSM_DEBUG_NONE 0
#define BSM_DEBUG_WITHHOLD_STAGE 1
#define BSM_DEBUG_CORRUPT_PATCH 2
int bsm_plan_debug(bsm_plan *plan, int what, int64_t arg);

/* Drop every cached plan of bsm_softmax / bsm_softmax_ex / bsm_softmax_ragged. */
void bsm_cache_clear(void);

/* ---- topology: the GB300 stand-in for cluster / memory-bank nearness ----
 * Sec. 2.1: a compute unit reaches its nearest memory bank with the least
 * latency.  On GB300 the "banks" are the two dies' L2 partitions and HBM
 * stacks.  The probe times dependent L2-hit loads from every SM to many
 * addresses, groups SMs whose latency profiles agree (one group per die), and
 * records the near and far latency (the weights of Sec. 4.2). */
typedef struct {
    int32_t device;
    int32_t n_sm;
    int32_t n_die;              /* 2 on GB300 when separable, else 1 */
    int32_t separable;          /* 1 if near/far latencies split cleanly */
    int8_t sm_die[BSM_MAX_SM];  /* die of SM id (%smid); -1 if never seen */
    int32_t sm_per_die[BSM_MAX_DIES];
    double l_near;              /* mean near L2-hit latency, SM cycles */
    double l_far;               /* mean far L2-hit latency, SM cycles */
    double separation;          /* mean |correlation| of SM profiles, 0..1 */
    int64_t granularity;        /* bytes of the smallest same-die address run seen */
    double probe_ms;
} bsm_topology;

/* Probe once per device (cached; force = 1 probes again).  Synchronous;
 * allocates and frees a 32 MiB scratch buffer.  device = -1: current. */
int bsm_topology_probe(int device, int force, bsm_topology *out);

/* Die of every `chunk`-byte chunk of the device buffer [ptr, ptr + bytes):
 * die_out (host, ceil(bytes/chunk) entries) gets the die whose L2 answers the
 * chunk's first line fastest.  chunk is a multiple of 128.  Reads the buffer,
 * writes nothing to it.  Needs a separable topology (else BSM_ERR_UNSUPPORTED).
 * Synchronous. */
int bsm_addr_die_map(int device, const void *ptr, int64_t bytes, int64_t chunk, int8_t *die_out);

/* The same map for a caller's grouping of the SMs instead of the probe's
 * dies: every chunk is timed from an SM of group 0 and one of group 1 and
 * goes to the faster group.  sm_group: host, BSM_MAX_SM entries indexed by
 * %smid, 0 or 1 (-1: the SM takes no part); both groups non-empty (else
 * BSM_ERR_INVALID_ARG).  For testing what the probe's grouping stands for.
 * Synchronous. */
int bsm_addr_group_map(int device, const void *ptr, int64_t bytes, int64_t chunk,
                       const int8_t *sm_group, int8_t *group_out);

/* Check of such a map (Sec. 4.1: a patch is "created" in the bank that holds
 * it): the SMs of each group read, once, only the chunk-byte chunks of
 * [ptr, ptr + bytes) that die_of_chunk (host, bytes / chunk entries of 0 or
 * 1) places on their group -- with invert != 0, only the others.  sm_group:
 * the SM grouping (as bsm_addr_group_map), or NULL for the probe's dies.
 * Run under a profiler, the L2's die-to-die (fabric) sector counters then say
 * how much of the traffic the map failed to keep on its die: none for a
 * right map and grouping, all of it inverted.  *xor_out gets the XOR of every
 * 32-bit word read (each chunk is read once, so it equals the XOR of the
 * whole buffer); *ms_out (may be NULL) the kernel's time.  bytes a multiple
 * of chunk, chunk of 16; ptr 16-byte aligned.  With sm_group NULL, needs a
 * separable topology (else BSM_ERR_UNSUPPORTED).  Synchronous; allocates and
 * frees small tables. */
int bsm_die_check_read(int device, const void *ptr, int64_t bytes, int64_t chunk,
                       const int8_t *die_of_chunk, const int8_t *sm_group, int invert,
                       uint32_t *xor_out, float *ms_out);

/* Raw probe matrix, for diagnostics: lat_out (host, BSM_MAX_SM x n_lines,
 * row = %smid) gets the mean cycles of a dependent L2-hit load from that SM to
 * byte offset line_off[i] of a 32 MiB scratch buffer (line_off multiples of
 * 128, below 32 MiB); seen_out[smid] = 1 for SMs that ran.  Synchronous. */
int bsm_probe_latency(int device, int32_t n_lines, const int64_t *line_off, int32_t reps,
                      float *lat_out, int32_t *seen_out);

/* ---- the scheduling steps alone, on the host (no GPU needed) ----
 * Runs the Sec. 4.1 table + overlap resolution and, when balance != 0, the
 * Sec. 4.2 load balance, on a caller-given address->bank map.  All arrays are
 * host memory owned by the caller. */
typedef struct {
    int32_t n_banks;            /* 1..BSM_MAX_DIES */
    int64_t n_patches;
    const int64_t *patch_begin; /* byte range [begin, end) of each patch */
    const int64_t *patch_end;
    int32_t n_maps;             /* 1 (input only) or 2 (input and output) */
    int64_t chunk[2];           /* bytes per map chunk */
    int64_t n_chunks[2];
    const int8_t *bank_of_chunk[2];
    uint64_t tie_seed;
    int32_t balance;            /* 0: CBMF only; 1: CBMF + load balance */
    const int32_t *units;       /* compute units near each bank */
    int64_t l_near, l_far;      /* latency weights (equal = unweighted) */
    const int64_t *cost;        /* work of each patch (bytes it moves) */
    int32_t method;             /* 0: Sec. 4.1 (+ 4.2 balance); 1: MINIMAX by longest
                                   patch first (uses the table, units, l_near, l_far) */
} bsm_schedule_desc;

typedef struct {
    int64_t *bytes_on_bank;     /* n_patches x n_banks */
    uint8_t *overlap;           /* n_patches */
    int64_t *N;                 /* n_banks */
    int32_t *bank;              /* n_patches: bank after overlap resolution */
    int64_t *L;                 /* n_banks */
    int32_t *queue_items;       /* n_patches: the banks' queues, concatenated */
    int64_t *queue_len;         /* n_banks */
    int32_t *moved;             /* n_patches: patch ids in the order moved */
    int64_t n_moved;
    int64_t *work_before;       /* n_banks: l_near*native + l_far*moved-in bytes */
    int64_t *work_after;        /* n_banks (MINIMAX: the cost assigned to each bank) */
} bsm_schedule_out;

int bsm_schedule_host(const bsm_schedule_desc *d, bsm_schedule_out *out);

/* ---- status ---- */

/* Sticky device-side status word of `device` (-1 = current), BSM_DEV_* bits
 * (the paper has no error reporting; the word is the contract's "device
 * faults are sticky" rule):
 * the library's own word OR-ed with the words of bsm_softmax_noalloc's fixed
 * array (so a timeout or bounds error there is not lost).  Synchronises the
 * device; allocates nothing.  bsm_device_status_clear zeroes both.  (The
 * contract's `int bsm_device_status(void)` gained the device and an output
 * argument, so that the status code and the bits travel separately.) */
int bsm_device_status(int device, uint32_t *status_out);
int bsm_device_status_clear(int device);

/* The 8-word device status block of `device` (-1 = current): word 0 is the
 * sticky BSM_DEV_* bits; when BSM_DEV_CHECK is set, words 1..7 describe the
 * first caught access (1 = kind: 1 shared read, 2 global store, 3 bulk copy,
 * 4 stage geometry; 2 = block; 3 = thread; 4..5 = offset, 6..7 = extent).
 * Synchronises the device. */
int bsm_device_debug(int device, uint32_t out[8]);

/* Select the self-checking kernel instantiation (on != 0) for launches made
 * after this call, in every thread: every shared-memory read, global store
 * and bulk copy is checked against its stage or buffer and skipped (and
 * recorded, see bsm_device_debug) when out of range.  Slower; for diagnosis. */
void bsm_set_device_checks(int on);

/* Name and description of the last CUDA runtime error a bsm call saw in this
 * thread ("" if none).  The string stays valid until the next bsm call in
 * the same thread. */
const char *bsm_last_cuda_error(void);

/* Largest row (C * element size) processed from a single shared-memory stage
 * on this device, bytes; longer rows take two passes (see Row length). */
int64_t bsm_max_row_bytes(int device);

/* Elements a ragged batch spans: max over the slices with rows[s] > 0 of
 * offsets[s] + rows[s] * cols[s] (0 for none), for a caller that checks its
 * buffers before bsm_softmax_ragged (the Python binding does).  Host only;
 * offsets/rows/cols: host arrays of n entries (NULL allowed when n == 0).
 * Returns -1 for n < 0, a NULL array, a negative offset or column count, or
 * an end past INT64_MAX. */
int64_t bsm_ragged_extent(int64_t n, const int64_t *offsets, const int32_t *rows, const int32_t *cols);

/* Static description of a status code. */
const char *bsm_status_string(int status);

/* Library version, (major << 16) | minor. */
int bsm_version(void);

#ifdef __cplusplus
}
#endif

#endif /* BSM_H */
