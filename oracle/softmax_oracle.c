/*
 * softmax_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, double-precision CPU oracle for the batched row-wise softmax
 * that "An optimal scheduling architecture for accelerating batch algorithms on
 * Neural Network processor architectures" (Nyshadham et al.) uses as its running
 * batch algorithm (Sec. 2: SOFTMAX on every 512 x 512 slice of a
 * (512*384) x 512 tensor; Sec. 6, SOFTMAX table).  The paper never writes the
 * formula down; the oracle uses the textbook definition along the last
 * dimension of each slice:
 *
 *     v[r,c] = x[r,c] + M[r,c]       (M = 0, or M = -inf where c > r under the
 *                                      causal flag; r is the row inside its slice)
 *     m_r    = max_c v[r,c]
 *     y[r,c] = exp(v[r,c] - m_r) / sum_c' exp(v[r,c'] - m_r)
 *
 * Subtracting m_r changes nothing mathematically (softmax is invariant to a
 * per-row shift); it only keeps exp() in range.  All arithmetic is IEEE double
 * on exactly-converted inputs, summed left to right, and rounded ONCE to the
 * output type with round-to-nearest-even.  Non-finite rows follow from the
 * same formula: a NaN or +inf anywhere in v, or a row that is all -inf, makes
 * the whole row NaN (0/0 or inf-inf).
 *
 * The backward pass (the paper's batch algorithms run "in the forward pass or
 * the backward pass", Sec. 1) is the vector-Jacobian product of the same
 * softmax: given y = softmax(v) and an upstream gradient dy of one row,
 *     dx[c] = y[c] * (dy[c] - sum_c' y[c'] * dy[c'])
 * in double, y and dy exactly converted, the dot product summed left to
 * right, rounded once to the output type.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg (and its
 * reference arm) may load this library.  It shares no code, header or constant
 * with the CUDA library: it has its own bf16 conversions, its own types and
 * its own thread pool.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_F32 0
#define ORC_BF16 1
#define ORC_CAUSAL 1u

/* bf16 is the upper half of an IEEE binary32: widening is a 16-bit shift. */
static double orc_bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest bf16 (8 significant bits, binary32 exponent
 * range, subnormals down to 2^-133), ties to even.  Written as "scale to an
 * integer grid, round with nearbyint (default mode = nearest-even), scale back",
 * which is exact because every scaling is by a power of two. */
uint16_t orc_double_to_bf16(double d)
{
    if (isnan(d))
        return (uint16_t)(signbit(d) ? 0xFFC0u : 0x7FC0u);
    uint16_t sign = signbit(d) ? 0x8000u : 0u;
    double a = fabs(d);
    if (a == 0.0)
        return sign;
    if (isinf(a))
        return (uint16_t)(sign | 0x7F80u);
    int e;
    frexp(a, &e);                  /* a in [2^(e-1), 2^e) */
    int q = e - 8;                 /* quantum of an 8-significant-bit number */
    if (q < -133)
        q = -133;                  /* bf16 subnormal spacing */
    double r = ldexp(nearbyint(ldexp(a, -q)), q);
    if (r >= 0x1p128)
        return (uint16_t)(sign | 0x7F80u);   /* rounds past the largest finite */
    float f = (float)r;            /* exact: r has <= 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(sign | (u >> 16));
}

static double orc_load(const void *x, int dtype, int64_t i)
{
    if (dtype == ORC_F32)
        return (double)((const float *)x)[i];
    return orc_bf16_to_double(((const uint16_t *)x)[i]);
}

/*
 * One row.  xrow points at the row's first element; row_in_slice is r (only
 * the causal mask uses it).  Writes the unrounded double result to y64 (may be
 * NULL) and the rounded result in the input dtype to yout (may be NULL).
 */
int orc_softmax_row(const void *xrow, int dtype, int64_t C, int64_t row_in_slice,
                    uint32_t flags, double *y64, void *yout)
{
    if (C <= 0 || (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    double *v = (double *)malloc((size_t)C * sizeof(double));
    if (!v)
        return -2;
    for (int64_t c = 0; c < C; ++c) {
        double mask = ((flags & ORC_CAUSAL) && c > row_in_slice) ? -INFINITY : 0.0;
        v[c] = orc_load(xrow, dtype, c) + mask;
    }
    double m = -INFINITY;
    for (int64_t c = 0; c < C; ++c)
        if (v[c] > m)
            m = v[c];
    double s = 0.0;
    for (int64_t c = 0; c < C; ++c)
        s += exp(v[c] - m);
    for (int64_t c = 0; c < C; ++c) {
        double yc = exp(v[c] - m) / s;
        if (y64)
            y64[c] = yc;
        if (yout) {
            if (dtype == ORC_F32)
                ((float *)yout)[c] = (float)yc;       /* C cast: round to nearest even */
            else
                ((uint16_t *)yout)[c] = orc_double_to_bf16(yc);
        }
    }
    free(v);
    return 0;
}

/* Backward of one row: y and dy point at the row's first elements. */
int orc_softmax_backward_row(const void *yrow, const void *dyrow, int dtype, int64_t C,
                             double *dx64, void *dxout)
{
    if (C <= 0 || (dtype != ORC_F32 && dtype != ORC_BF16))
        return -1;
    double dot = 0.0;
    for (int64_t c = 0; c < C; ++c)
        dot += orc_load(yrow, dtype, c) * orc_load(dyrow, dtype, c);
    for (int64_t c = 0; c < C; ++c) {
        double d = orc_load(yrow, dtype, c) * (orc_load(dyrow, dtype, c) - dot);
        if (dx64)
            dx64[c] = d;
        if (dxout) {
            if (dtype == ORC_F32)
                ((float *)dxout)[c] = (float)d;
            else
                ((uint16_t *)dxout)[c] = orc_double_to_bf16(d);
        }
    }
    return 0;
}

/* ---- batched form: slices s = 0..B-1, slice s has rows[s] x cols[s] elements
 *      starting at element offsets[s] of x (and of y64 / yout). ---- */

typedef struct {
    const void *x;
    const void *dy;            /* backward: upstream gradient (x is y) */
    int dtype;
    int64_t nslices;
    const int64_t *offsets;
    const int32_t *rows;
    const int32_t *cols;
    uint32_t flags;
    double *y64;
    void *yout;
    int64_t total_rows;
    const int64_t *row_base;   /* prefix sums of rows[] */
    int nthreads;
    int tid;
    int status;
} orc_job;

static int64_t orc_find_slice(const int64_t *row_base, int64_t nslices, int64_t g)
{
    int64_t lo = 0, hi = nslices - 1;
    while (lo < hi) {
        int64_t mid = (lo + hi + 1) / 2;
        if (row_base[mid] <= g)
            lo = mid;
        else
            hi = mid - 1;
    }
    return lo;
}

static void *orc_worker(void *arg)
{
    orc_job *j = (orc_job *)arg;
    size_t es = j->dtype == ORC_F32 ? 4 : 2;
    /* contiguous block of global rows per thread */
    int64_t per = (j->total_rows + j->nthreads - 1) / j->nthreads;
    int64_t g0 = per * j->tid, g1 = g0 + per;
    if (g1 > j->total_rows)
        g1 = j->total_rows;
    for (int64_t g = g0; g < g1; ++g) {
        int64_t s = orc_find_slice(j->row_base, j->nslices, g);
        int64_t r = g - j->row_base[s];
        int64_t C = j->cols[s];
        int64_t e = j->offsets[s] + r * C;
        int rc;
        if (j->dy)
            rc = orc_softmax_backward_row((const char *)j->x + e * es, (const char *)j->dy + e * es,
                                          j->dtype, C, j->y64 ? j->y64 + e : NULL,
                                          j->yout ? (void *)((char *)j->yout + e * es) : NULL);
        else
            rc = orc_softmax_row((const char *)j->x + e * es, j->dtype, C, r, j->flags,
                                 j->y64 ? j->y64 + e : NULL,
                                 j->yout ? (void *)((char *)j->yout + e * es) : NULL);
        if (rc) {
            j->status = rc;
            break;
        }
    }
    return NULL;
}

static int orc_run_batched(const void *x, const void *dy, int dtype, int64_t nslices,
                           const int64_t *offsets, const int32_t *rows, const int32_t *cols,
                           uint32_t flags, double *y64, void *yout, int nthreads)
{
    if (nslices < 0 || (nslices > 0 && (!x || !offsets || !rows || !cols)))
        return -1;
    if (nslices == 0)
        return 0;
    if (nthreads < 1)
        nthreads = 1;
    int64_t *row_base = (int64_t *)malloc((size_t)(nslices + 1) * sizeof(int64_t));
    if (!row_base)
        return -2;
    row_base[0] = 0;
    for (int64_t s = 0; s < nslices; ++s) {
        if (rows[s] < 0 || cols[s] <= 0) {
            free(row_base);
            return -1;
        }
        row_base[s + 1] = row_base[s] + rows[s];
    }
    int64_t total = row_base[nslices];
    if ((int64_t)nthreads > total)
        nthreads = total > 0 ? (int)total : 1;
    orc_job *jobs = (orc_job *)calloc((size_t)nthreads, sizeof(orc_job));
    pthread_t *th = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
    if (!jobs || !th) {
        free(row_base);
        free(jobs);
        free(th);
        return -2;
    }
    for (int t = 0; t < nthreads; ++t) {
        orc_job j = {x, dy, dtype, nslices, offsets, rows, cols, flags, y64, yout,
                     total, row_base, nthreads, t, 0};
        jobs[t] = j;
    }
    int status = 0;
    for (int t = 1; t < nthreads; ++t)
        if (pthread_create(&th[t], NULL, orc_worker, &jobs[t]))
            jobs[t].status = -3;
    orc_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t)
        if (jobs[t].status != -3)
            pthread_join(th[t], NULL);
    for (int t = 0; t < nthreads; ++t)
        if (jobs[t].status)
            status = jobs[t].status;
    free(row_base);
    free(jobs);
    free(th);
    return status;
}

int orc_softmax_batched(const void *x, int dtype, int64_t nslices, const int64_t *offsets,
                        const int32_t *rows, const int32_t *cols, uint32_t flags,
                        double *y64, void *yout, int nthreads)
{
    return orc_run_batched(x, NULL, dtype, nslices, offsets, rows, cols, flags, y64, yout, nthreads);
}

/* Backward over every slice: y and dy laid out like the forward's x. */
int orc_softmax_backward_batched(const void *y, const void *dy, int dtype, int64_t nslices,
                                 const int64_t *offsets, const int32_t *rows, const int32_t *cols,
                                 double *dx64, void *dxout, int nthreads)
{
    if (nslices > 0 && !dy)
        return -1;
    return orc_run_batched(y, dy, dtype, nslices, offsets, rows, cols, 0u, dx64, dxout, nthreads);
}
