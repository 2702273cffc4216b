/*
 * Seeded synthetic inputs shared by the oracle side and the CUDA side.
 *
 * This file draws random numbers and nothing else: it holds none of the decoder-layer arithmetic.
 * Every value is a pure function of (seed, element index), so the result does not depend on the
 * number of threads that fill an array.
 *
 * Generator: SplitMix64 (G. Steele, D. Lea, C. Flood, "Fast Splittable Pseudorandom Number
 * Generators", OOPSLA 2014) used in counter mode: word i of stream `seed` is
 * mix(key(seed) + (i + 1) * GAMMA).  Normal variates come from the Box-Muller transform
 * (G. Box, M. Muller, 1958) applied to consecutive pairs of words.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>

#define SYNTH_GAMMA 0x9e3779b97f4a7c15ULL

static inline uint64_t synth_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

static inline uint64_t synth_word(uint64_t key, uint64_t i) {
    return synth_mix(key + (i + 1) * SYNTH_GAMMA);
}

static inline uint64_t synth_key(uint64_t seed) { return synth_mix(seed ^ 0x5851f42d4c957f2dULL); }

/* Raw 64-bit words, for tests of the generator itself. */
void synth_words(uint64_t* out, int64_t n, uint64_t seed) {
    const uint64_t key = synth_key(seed);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = synth_word(key, (uint64_t)i);
}

/* Standard normal variate number i of stream `key` (Box-Muller on words 2k and 2k+1). */
static inline double synth_normal_at(uint64_t key, int64_t i) {
    const uint64_t k = (uint64_t)(i >> 1);
    const uint64_t a = synth_word(key, 2 * k);
    const uint64_t b = synth_word(key, 2 * k + 1);
    const double u1 = ((double)(a >> 11) + 1.0) * 0x1.0p-53; /* (0, 1] */
    const double u2 = (double)(b >> 11) * 0x1.0p-53;         /* [0, 1) */
    const double r = sqrt(-2.0 * log(u1));
    const double t = 6.283185307179586476925286766559 * u2;
    return (i & 1) ? r * sin(t) : r * cos(t);
}

/* out[i] = fp16(fp32(mean + std * N_i)), rounded to nearest even at each narrowing. */
void synth_normal_f16(uint16_t* out, int64_t n, uint64_t seed, double mean, double std) {
    const uint64_t key = synth_key(seed);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        const float v = (float)(mean + std * synth_normal_at(key, i));
        const _Float16 h = (_Float16)v;
        uint16_t bits;
        __builtin_memcpy(&bits, &h, sizeof bits);
        out[i] = bits;
    }
}

/* out[i] = fp32(mean + std * N_i). */
void synth_normal_f32(float* out, int64_t n, uint64_t seed, double mean, double std) {
    const uint64_t key = synth_key(seed);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = (float)(mean + std * synth_normal_at(key, i));
}

/* out[i] uniform in [lo, hi) (multiply-shift on the top 32 bits of each word). */
void synth_uniform_i32(int32_t* out, int64_t n, uint64_t seed, int32_t lo, int32_t hi) {
    const uint64_t key = synth_key(seed);
    const uint64_t range = (uint64_t)((int64_t)hi - (int64_t)lo);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        const uint64_t w = synth_word(key, (uint64_t)i) >> 32;
        out[i] = (int32_t)((int64_t)lo + (int64_t)((w * range) >> 32));
    }
}
