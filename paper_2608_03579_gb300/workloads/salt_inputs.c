/*
 * Seeded synthetic inputs for the SALT serving path.
 *
 * Counter-based generation: element i of a (seed, stream) sequence is the
 * (i+1)-th output of SplitMix64 (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) started from a per-stream
 * state, so any element can be produced on its own and in any order.
 * Normal deviates come from the Box-Muller transform (Box and Muller, 1958)
 * applied to consecutive pairs of uniforms, then rounded to bf16
 * (binary32 round-to-nearest-even, then round-to-nearest-even of the low
 * 16 bits).
 *
 * This file draws inputs and nothing else: none of the method's arithmetic
 * is here.  Both the oracle side and the CUDA side read the arrays it fills.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>

#define SI_GOLDEN 0x9E3779B97F4A7C15ULL

static uint64_t si_mix(uint64_t z)
{
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

/* Per-stream starting state. */
static uint64_t si_base(uint64_t seed, uint64_t stream)
{
    return si_mix(seed ^ si_mix(stream ^ 0xD1B54A32D192ED03ULL));
}

/* Element i of the stream: the (i+1)-th SplitMix64 output from base. */
static uint64_t si_bits(uint64_t base, uint64_t i)
{
    return si_mix(base + (i + 1) * SI_GOLDEN);
}

uint64_t salt_inputs_bits(uint64_t seed, uint64_t stream, uint64_t i)
{
    return si_bits(si_base(seed, stream), i);
}

/* Uniform on [0, 1) with 53 random bits. */
static double si_unit(uint64_t b)
{
    return (double)(b >> 11) * (1.0 / 9007199254740992.0);
}

static uint16_t si_bf16_from_float(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u) /* inf / nan: keep the top half */
        return (uint16_t)(u >> 16);
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* Standard normal deviate number i of the stream (Box-Muller pair i/2). */
static double si_normal(uint64_t base, uint64_t i)
{
    uint64_t pair = i >> 1;
    double u1 = 1.0 - si_unit(si_bits(base, 2 * pair)); /* (0, 1] */
    double u2 = si_unit(si_bits(base, 2 * pair + 1));   /* [0, 1) */
    double r = sqrt(-2.0 * log(u1));
    double th = 6.283185307179586476925286766559 * u2;
    return (i & 1) ? r * sin(th) : r * cos(th);
}

typedef struct {
    uint64_t base, first;
    int64_t lo, hi;
    double sigma;
    uint16_t *out;
} si_job;

static void *si_normal_worker(void *p)
{
    si_job *j = (si_job *)p;
    for (int64_t k = j->lo; k < j->hi; ++k) {
        double v = j->sigma * si_normal(j->base, j->first + (uint64_t)k);
        j->out[k] = si_bf16_from_float((float)v);
    }
    return NULL;
}

/* out[k] = bf16(sigma * N(seed, stream, first + k)), k in [0, n). */
void salt_inputs_normal_bf16(uint64_t seed, uint64_t stream, uint64_t first, int64_t n,
                             double sigma, uint16_t *out, int n_threads)
{
    uint64_t base = si_base(seed, stream);
    if (n_threads < 1) n_threads = 1;
    if (n_threads > 64) n_threads = 64;
    if (n < (int64_t)1 << 16) n_threads = 1;
    if (n_threads == 1) {
        si_job j = {base, first, 0, n, sigma, out};
        si_normal_worker(&j);
        return;
    }
    pthread_t th[64];
    int created[64];
    si_job jobs[64];
    for (int t = 0; t < n_threads; ++t) {
        jobs[t].base = base;
        jobs[t].first = first;
        jobs[t].lo = n * t / n_threads;
        jobs[t].hi = n * (t + 1) / n_threads;
        jobs[t].sigma = sigma;
        jobs[t].out = out;
        created[t] = pthread_create(&th[t], NULL, si_normal_worker, &jobs[t]) == 0;
        if (!created[t]) si_normal_worker(&jobs[t]);
    }
    for (int t = 0; t < n_threads; ++t)
        if (created[t]) pthread_join(th[t], NULL);
}

/* out[k] = uniform [0, 1) number first + k of the stream. */
void salt_inputs_uniform(uint64_t seed, uint64_t stream, uint64_t first, int64_t n, double *out)
{
    uint64_t base = si_base(seed, stream);
    for (int64_t k = 0; k < n; ++k)
        out[k] = si_unit(si_bits(base, first + (uint64_t)k));
}
