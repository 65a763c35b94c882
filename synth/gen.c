/*
 * Seeded synthetic-input generator shared by the fp64 oracle and the GPU path.
 *
 * It holds none of the decoder's arithmetic: it only turns (seed, stream,
 * element index) into numbers.  Every value is a pure function of those three
 * integers, so the output is identical for any thread count and for any
 * sub-range requested through `offset`.
 *
 * Generator: SplitMix64 (Steele, Lea, Flood, "Fast splittable pseudorandom
 * number generators", OOPSLA 2014), used counter-style: the i-th draw of a
 * stream is the SplitMix64 output for state key + (i + 1) * golden-gamma.
 * Normals: Box-Muller (1958), one normal per pair of draws (the cosine
 * branch), computed in double precision.
 * bf16: the double is rounded to float (C cast, round-to-nearest-even), then
 * the float to bf16 by round-to-nearest-even on its bit pattern.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <string.h>
#include <unistd.h>

#define SYNTH_GOLDEN 0x9E3779B97F4A7C15ULL
#define SYNTH_STREAM_MUL 0xD1B54A32D192ED03ULL
#define SYNTH_TWO_PI 6.283185307179586476925286766559

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t stream_key(uint64_t seed, uint64_t stream) {
    return mix64(seed * SYNTH_GOLDEN + SYNTH_GOLDEN) ^ mix64((stream + 1) * SYNTH_STREAM_MUL);
}

static inline uint64_t draw(uint64_t key, uint64_t ctr) {
    return mix64(key + (ctr + 1) * SYNTH_GOLDEN);
}

/* Standard normal for element i of the stream. */
static inline double normal_at(uint64_t key, uint64_t i) {
    uint64_t a = draw(key, 2 * i), b = draw(key, 2 * i + 1);
    double u1 = (double)((a >> 11) + 1) * 0x1.0p-53; /* (0, 1] */
    double u2 = (double)(b >> 11) * 0x1.0p-53;       /* [0, 1) */
    return sqrt(-2.0 * log(u1)) * cos(SYNTH_TWO_PI * u2);
}

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

enum { KIND_BF16 = 0, KIND_F32 = 1, KIND_I32 = 2 };

typedef struct {
    int kind;
    uint64_t key, offset, begin, end;
    double mean, sigma;
    int32_t lo, hi;
    void* out;
} job_t;

static void* run_job(void* arg) {
    job_t* j = (job_t*)arg;
    for (uint64_t i = j->begin; i < j->end; ++i) {
        uint64_t g = j->offset + i;
        if (j->kind == KIND_I32) {
            uint64_t span = (uint64_t)((int64_t)j->hi - (int64_t)j->lo);
            uint64_t r = draw(j->key, g) >> 32;
            ((int32_t*)j->out)[i] = (int32_t)((int64_t)j->lo + (int64_t)((r * span) >> 32));
        } else {
            double v = j->mean + j->sigma * normal_at(j->key, g);
            if (j->kind == KIND_F32)
                ((float*)j->out)[i] = (float)v;
            else
                ((uint16_t*)j->out)[i] = f32_to_bf16_rne((float)v);
        }
    }
    return NULL;
}

static int run(job_t proto, uint64_t n, int nthreads) {
    if (nthreads <= 0) {
        long c = sysconf(_SC_NPROCESSORS_ONLN);
        nthreads = c > 0 ? (int)c : 1;
    }
    if (nthreads > 256) nthreads = 256;
    uint64_t min_chunk = 1u << 16;
    if ((uint64_t)nthreads * min_chunk > n) nthreads = (int)((n + min_chunk - 1) / min_chunk);
    if (nthreads < 1) nthreads = 1;
    pthread_t th[256];
    job_t jobs[256];
    uint64_t per = (n + (uint64_t)nthreads - 1) / (uint64_t)nthreads;
    int started = 0;
    for (int t = 0; t < nthreads; ++t) {
        jobs[t] = proto;
        jobs[t].begin = (uint64_t)t * per;
        jobs[t].end = jobs[t].begin + per > n ? n : jobs[t].begin + per;
        if (jobs[t].begin >= jobs[t].end) break;
        if (t == 0) continue; /* the calling thread runs chunk 0 */
        if (pthread_create(&th[t], NULL, run_job, &jobs[t]) != 0) {
            run_job(&jobs[t]);
            jobs[t].end = jobs[t].begin; /* mark as done inline */
            th[t] = 0;
        }
        started = t;
    }
    if (n > 0) run_job(&jobs[0]);
    for (int t = 1; t <= started; ++t)
        if (jobs[t].end > jobs[t].begin) pthread_join(th[t], NULL);
    return 0;
}

int synth_normal_bf16(uint64_t seed, uint64_t stream, uint64_t offset, uint64_t n, double mean,
                      double sigma, uint16_t* out, int nthreads) {
    job_t p = {KIND_BF16, stream_key(seed, stream), offset, 0, 0, mean, sigma, 0, 0, out};
    return run(p, n, nthreads);
}

int synth_normal_f32(uint64_t seed, uint64_t stream, uint64_t offset, uint64_t n, double mean,
                     double sigma, float* out, int nthreads) {
    job_t p = {KIND_F32, stream_key(seed, stream), offset, 0, 0, mean, sigma, 0, 0, out};
    return run(p, n, nthreads);
}

/* Uniform integers in [lo, hi): the top 32 bits of each draw scaled by (hi - lo). */
int synth_uniform_i32(uint64_t seed, uint64_t stream, uint64_t offset, uint64_t n, int32_t lo,
                      int32_t hi, int32_t* out, int nthreads) {
    if (hi <= lo) return -1;
    job_t p = {KIND_I32, stream_key(seed, stream), offset, 0, 0, 0.0, 0.0, lo, hi, out};
    return run(p, n, nthreads);
}

/* Raw SplitMix64 draw, exported so tests can check the generator against its definition. */
uint64_t synth_raw_draw(uint64_t seed, uint64_t stream, uint64_t ctr) {
    return draw(stream_key(seed, stream), ctr);
}
