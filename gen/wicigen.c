/*
 * Seeded synthetic inputs for the batch-1 decoder forward pass: bf16 weight
 * tensors and uniform-random prompt token ids.  This file holds none of the
 * model's arithmetic; both the CPU oracle and the CUDA path consume the bytes
 * it writes, so the two never need a common random-number library.
 *
 * Generator (its own definition, stated once):
 *   mix64(z)          the splitmix64 output function (Steele, Lea & Flood,
 *                     "Fast splittable pseudorandom number generators",
 *                     OOPSLA 2014; constants as in Vigna's public splitmix64).
 *   draw(key, i)      = mix64(key + (i + 1) * GAMMA): the i-th output of a
 *                     splitmix64 stream started at state `key`.
 *   stream(seed, tag) = mix64((seed << 32) ^ tag), one stream per tensor.
 *   normal element e  uses draws 3e, 3e+1, 3e+2 = twelve 16-bit fields b_k;
 *                     s = sum_k (b_k + 1/2)/65536 - 6 (sum of twelve
 *                     uniforms, an approximately N(0,1) variate).  The
 *                     numerator sum_k b_k + 6 - 393216 is an exact integer,
 *                     so s is exact in double and the value is
 *                     bf16_rne((float)(s * std)) on any IEEE-754 machine.
 *   token i           = draw(stream(seed, PROMPT_TAG), i) mod vocab.
 *
 * Built with -ffp-contract=off so no multiply-add is fused.
 */
#include <stdint.h>
#include <string.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

uint64_t wicigen_draw(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GAMMA); }

uint64_t wicigen_stream(uint64_t seed, uint64_t tag) { return mix64((seed << 32) ^ tag); }

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return 0x7FC0; /* NaN */
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static inline double normal_at(uint64_t key, uint64_t e) {
    int64_t acc = 0;
    for (int j = 0; j < 3; ++j) {
        uint64_t r = wicigen_draw(key, 3 * e + (uint64_t)j);
        acc += (int64_t)(r & 0xFFFF) + (int64_t)((r >> 16) & 0xFFFF) +
               (int64_t)((r >> 32) & 0xFFFF) + (int64_t)(r >> 48);
    }
    return (double)(acc + 6 - 393216) / 65536.0;
}

/* out[e] = bf16 bits of N(0, std) sample e of stream(seed, tag), e in [e0, e0+n). */
void wicigen_normal_bf16(uint64_t seed, uint64_t tag, double std, uint64_t e0, uint64_t n,
                         uint16_t *out) {
    const uint64_t key = wicigen_stream(seed, tag);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) {
        double s = normal_at(key, e0 + (uint64_t)i) * std;
        out[i] = f32_to_bf16_rne((float)s);
    }
}

/* out[e] = bf16 bits of 1 + std * s_e (norm gains that are not all one), same stream rule. */
void wicigen_gain_bf16(uint64_t seed, uint64_t tag, double std, uint64_t e0, uint64_t n, uint16_t *out) {
    const uint64_t key = wicigen_stream(seed, tag);
    for (uint64_t i = 0; i < n; ++i) out[i] = f32_to_bf16_rne((float)(1.0 + normal_at(key, e0 + i) * std));
}

/* out[e] = the same approximately-normal variates as doubles (for statistics tests). */
void wicigen_normal_f64(uint64_t seed, uint64_t tag, uint64_t e0, uint64_t n, double *out) {
    const uint64_t key = wicigen_stream(seed, tag);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < (int64_t)n; ++i) out[i] = normal_at(key, e0 + (uint64_t)i);
}

/* out[i] = draw(stream(seed, tag), i) mod vocab, i in [0, n). */
void wicigen_tokens(uint64_t seed, uint64_t tag, uint64_t vocab, uint64_t n, int32_t *out) {
    const uint64_t key = wicigen_stream(seed, tag);
    for (uint64_t i = 0; i < n; ++i) out[i] = (int32_t)(wicigen_draw(key, i) % vocab);
}

/* out[i] = bf16 bits of `value` (norm gains are constant). */
void wicigen_fill_bf16(float value, uint64_t n, uint16_t *out) {
    const uint16_t b = f32_to_bf16_rne(value);
    for (uint64_t i = 0; i < n; ++i) out[i] = b;
}
