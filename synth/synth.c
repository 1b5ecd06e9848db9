/*
 * Seeded synthetic input generator: weights, prompts and calibration token
 * streams for the early-exit decode workloads.
 *
 * This file produces INPUT DATA only. It holds none of the decode method's
 * arithmetic and is shared, as data, by the CPU oracle and the CUDA path.
 *
 * Generator: SplitMix64 (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) used as a counter-based
 * stream.  A stream is named by (seed, stream id); its n-th 64-bit output is
 *     key    = mix(seed XOR (sid * 0xD1B54A32D192ED03))
 *     out(n) = mix(key + (n + 1) * 0x9E3779B97F4A7C15)
 * with mix() the SplitMix64 finaliser.  Normal variates use the Box-Muller
 * transform (cosine branch) in double precision: element i of a tensor takes
 * outputs 2i and 2i+1,
 *     u1 = ((out(2i)   >> 11) + 1) * 2^-53     in (0, 1]
 *     u2 =  (out(2i+1) >> 11)      * 2^-53     in [0, 1)
 *     n  = sqrt(-2 ln u1) * cos(2 pi u2)
 * and the stored value is bf16(float(n * std)), rounded to nearest even.
 * Token ids are out(n) mod V.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t sm64_mix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

static inline uint64_t sm64_key(uint64_t seed, uint64_t sid) {
    return sm64_mix(seed ^ (sid * 0xD1B54A32D192ED03ULL));
}

static inline uint64_t sm64_at(uint64_t key, uint64_t n) {
    return sm64_mix(key + (n + 1) * 0x9E3779B97F4A7C15ULL);
}

/* float -> bf16 bits, round to nearest even (NaN kept quiet). */
static inline uint16_t synth_f32_to_bf16(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    if ((u & 0x7f800000u) == 0x7f800000u) {
        if (u & 0x007fffffu) return (uint16_t)((u >> 16) | 0x0040u);
        return (uint16_t)(u >> 16);
    }
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/* Raw 64-bit outputs [first, first + n) of stream (seed, sid). */
void synth_u64(uint64_t seed, uint64_t sid, uint64_t first, int64_t n, uint64_t* out) {
    const uint64_t key = sm64_key(seed, sid);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = sm64_at(key, first + (uint64_t)i);
}

/* n bf16 values N(mean, std^2) from stream (seed, sid). */
void synth_normal_bf16(uint64_t seed, uint64_t sid, int64_t n, double mean, double std,
                       uint16_t* out) {
    const uint64_t key = sm64_key(seed, sid);
    const double two_pi = 6.283185307179586476925286766559;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        const uint64_t a = sm64_at(key, 2 * (uint64_t)i);
        const uint64_t b = sm64_at(key, 2 * (uint64_t)i + 1);
        const double u1 = (double)((a >> 11) + 1) * 0x1.0p-53;
        const double u2 = (double)(b >> 11) * 0x1.0p-53;
        const double z = sqrt(-2.0 * log(u1)) * cos(two_pi * u2);
        out[i] = synth_f32_to_bf16((float)(mean + z * std));
    }
}

/* n bf16 values: value on the diagonal of a rows x cols matrix is
 * 1 + N(0, std^2), off-diagonal N(0, std^2).  Used for readout matrices
 * initialised near the identity. */
void synth_identity_plus_normal_bf16(uint64_t seed, uint64_t sid, int64_t rows, int64_t cols,
                                     double std, uint16_t* out) {
    const uint64_t key = sm64_key(seed, sid);
    const double two_pi = 6.283185307179586476925286766559;
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < rows * cols; ++i) {
        const uint64_t a = sm64_at(key, 2 * (uint64_t)i);
        const uint64_t b = sm64_at(key, 2 * (uint64_t)i + 1);
        const double u1 = (double)((a >> 11) + 1) * 0x1.0p-53;
        const double u2 = (double)(b >> 11) * 0x1.0p-53;
        const double z = sqrt(-2.0 * log(u1)) * cos(two_pi * u2) * std;
        const double diag = ((i / cols) == (i % cols)) ? 1.0 : 0.0;
        out[i] = synth_f32_to_bf16((float)(diag + z));
    }
}

/* n bf16 copies of one value. */
void synth_fill_bf16(int64_t n, double value, uint16_t* out) {
    const uint16_t v = synth_f32_to_bf16((float)value);
    for (int64_t i = 0; i < n; ++i) out[i] = v;
}

/* n token ids uniform on [0, vocab) (modulo bias below 1e-13 for vocab < 2^21). */
void synth_token_ids(uint64_t seed, uint64_t sid, int64_t n, int32_t vocab, int32_t* out) {
    const uint64_t key = sm64_key(seed, sid);
    for (int64_t i = 0; i < n; ++i) out[i] = (int32_t)(sm64_at(key, (uint64_t)i) % (uint64_t)vocab);
}

/* n Bernoulli(rate) draws (1 with probability rate). */
void synth_bernoulli(uint64_t seed, uint64_t sid, int64_t n, double rate, int8_t* out) {
    const uint64_t key = sm64_key(seed, sid);
    for (int64_t i = 0; i < n; ++i) {
        const double u = (double)(sm64_at(key, (uint64_t)i) >> 11) * 0x1.0p-53;
        out[i] = (int8_t)(u < rate ? 1 : 0);
    }
}
