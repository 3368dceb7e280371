/*
 * gen.c -- seeded synthetic inputs for the batched softmax.
 *
 * This module holds no softmax or scheduling arithmetic: it only makes input
 * numbers and shapes.  Both the CUDA path (through the tests and the bench)
 * and the CPU oracle consume the host bytes it writes.
 *
 * Counter-based: value k depends only on (seed, k), so the fill is split over
 * threads without changing a single bit.  The uniform source is splitmix64
 * (Steele, Lea and Flood, "Fast splittable pseudorandom number generators",
 * 2014; constants as published by Vigna): draw i is the mix of
 * seed + (i + 1) * golden-gamma.  Normals come from the Box-Muller transform
 * (pair k uses draws 2k and 2k+1; element 2k takes the cosine branch, element
 * 2k+1 the sine branch), in double, then scaled by sigma and rounded to the
 * element type: float32 by the C conversion (round to nearest even), bf16 by
 * rounding that float32 to nearest even on its upper 16 bits.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>

#define GEN_F32 0
#define GEN_BF16 1

static inline uint64_t gen_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

uint64_t gen_splitmix64(uint64_t seed, uint64_t i)
{
    return gen_mix(seed + (i + 1) * 0x9E3779B97F4A7C15ULL);
}

/* uniform in (0, 1]: 53 random bits, offset by one so log() never sees 0 */
static inline double gen_unit(uint64_t seed, uint64_t i)
{
    return (double)((gen_splitmix64(seed, i) >> 11) + 1) * 0x1p-53;
}

double gen_normal(uint64_t seed, uint64_t k)
{
    uint64_t pair = k >> 1;
    double u1 = gen_unit(seed, 2 * pair), u2 = gen_unit(seed, 2 * pair + 1);
    double r = sqrt(-2.0 * log(u1));
    double t = 6.283185307179586 * u2;
    return (k & 1) ? r * sin(t) : r * cos(t);
}

static uint16_t gen_f32_to_bf16(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu))
        return (uint16_t)((u >> 16) | 0x0040u);   /* quiet NaN */
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

typedef struct {
    void *out;
    int dtype;
    uint64_t seed;
    double sigma, mu;
    int64_t first, count;     /* element range written by this worker */
    int64_t index_base;       /* draw index of element 0 of `out` */
} gen_job;

static void *gen_worker(void *arg)
{
    gen_job *j = (gen_job *)arg;
    for (int64_t e = j->first; e < j->first + j->count; ++e) {
        double v = j->mu + j->sigma * gen_normal(j->seed, (uint64_t)(j->index_base + e));
        float f = (float)v;
        if (j->dtype == GEN_F32)
            ((float *)j->out)[e] = f;
        else
            ((uint16_t *)j->out)[e] = gen_f32_to_bf16(f);
    }
    return NULL;
}

/* Fill out[0..n) with mu + sigma * N(0,1) draws index_base .. index_base+n-1. */
int gen_fill_normal(void *out, int dtype, int64_t n, uint64_t seed, double mu, double sigma,
                    int64_t index_base, int nthreads)
{
    if (n < 0 || (n > 0 && !out) || (dtype != GEN_F32 && dtype != GEN_BF16))
        return -1;
    if (nthreads < 1)
        nthreads = 1;
    if (nthreads > 256)
        nthreads = 256;
    if ((int64_t)nthreads > n / 65536 + 1)
        nthreads = (int)(n / 65536 + 1);
    gen_job jobs[256];
    pthread_t th[256];
    int64_t per = (n + nthreads - 1) / nthreads;
    for (int t = 0; t < nthreads; ++t) {
        int64_t f = per * t, c = per;
        if (f > n)
            f = n;
        if (f + c > n)
            c = n - f;
        gen_job j = {out, dtype, seed, sigma, mu, f, c, index_base};
        jobs[t] = j;
    }
    int started[256] = {0};
    for (int t = 1; t < nthreads; ++t)
        started[t] = pthread_create(&th[t], NULL, gen_worker, &jobs[t]) == 0;
    gen_worker(&jobs[0]);
    for (int t = 1; t < nthreads; ++t) {
        if (started[t])
            pthread_join(th[t], NULL);
        else
            gen_worker(&jobs[t]);
    }
    return 0;
}

/* Ragged shapes: slice s has rows = row_unit * (1 + d % row_steps) and
 * cols = col_unit * (1 + d' % col_steps), d = draw 2s, d' = draw 2s+1 of the
 * shape stream. */
int gen_ragged_shapes(int32_t *rows, int32_t *cols, int64_t nslices, uint64_t shape_seed,
                      int32_t row_unit, int32_t row_steps, int32_t col_unit, int32_t col_steps)
{
    if (nslices < 0 || row_steps < 1 || col_steps < 1)
        return -1;
    for (int64_t s = 0; s < nslices; ++s) {
        rows[s] = row_unit * (int32_t)(1 + gen_splitmix64(shape_seed, 2 * (uint64_t)s) % (uint64_t)row_steps);
        cols[s] = col_unit * (int32_t)(1 + gen_splitmix64(shape_seed, 2 * (uint64_t)s + 1) % (uint64_t)col_steps);
    }
    return 0;
}
