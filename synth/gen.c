/*
 * Seeded synthetic-input generator shared by the CPU oracle's tests and the
 * GPU path's tests and benchmark.  It holds none of the draft model's
 * arithmetic: it only turns (seed, tag, index) into numbers.
 *
 * Counter-based stream.  For a tensor with 64-bit seed `seed` and 64-bit tag
 * `tag`, the generator state is s0 = mix(seed ^ mix(tag ^ TAG_SALT)) and the
 * i-th raw 64-bit output is mix(s0 + (i + 1) * GAMMA), which is exactly the
 * i-th output of SplitMix64 (Steele, Lea and Flood, "Fast splittable
 * pseudorandom number generators", OOPSLA 2014) started from state s0.
 * Every element therefore depends only on (seed, tag, index): any slice can be
 * generated on its own and in parallel, with identical bits on every machine
 * (integer arithmetic plus correctly rounded IEEE-754 double operations).
 *
 * Normal-shaped draws use the Irwin-Hall construction: eight 16-bit uniform
 * integers (taken from two raw outputs) are summed exactly, centred and scaled
 * to the requested standard deviation.  Mean and variance match N(0, sigma^2);
 * the support is cut at about 4.9 sigma.
 */
#include <stdint.h>
#include <string.h>
#include <math.h>

#define GAMMA 0x9e3779b97f4a7c15ULL
#define TAG_SALT 0x5851f42d4c957f2dULL

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ULL;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebULL;
    return z ^ (z >> 31);
}

static inline uint64_t stream_base(uint64_t seed, uint64_t tag) {
    return mix64(seed ^ mix64(tag ^ TAG_SALT));
}

static inline uint64_t raw_at(uint64_t s0, uint64_t i) {
    return mix64(s0 + (i + 1) * GAMMA);
}

/* Plain SplitMix64 step, exposed so tests can check it against the published
 * reference outputs. */
uint64_t synth_splitmix64_next(uint64_t *state) {
    *state += GAMMA;
    return mix64(*state);
}

uint64_t synth_raw(uint64_t seed, uint64_t tag, uint64_t i) {
    return raw_at(stream_base(seed, tag), i);
}

/* Irwin-Hall(8) of 16-bit uniforms: S in [0, 8*65535], mean 262140,
 * variance 8*(65536^2-1)/12. */
static inline double irwin_hall8(uint64_t s0, uint64_t i, double scale) {
    uint64_t a = raw_at(s0, 2 * i), b = raw_at(s0, 2 * i + 1);
    int64_t s = 0;
    for (int q = 0; q < 4; ++q) {
        s += (int64_t)((a >> (16 * q)) & 0xFFFFu);
        s += (int64_t)((b >> (16 * q)) & 0xFFFFu);
    }
    return (double)(s - 262140) * scale;
}

static double ih8_scale(double sigma) {
    /* 1 / std of the centred sum.  IEEE-754 sqrt and division are correctly
     * rounded, so the constant is identical on every conforming machine. */
    double var = 8.0 * (65536.0 * 65536.0 - 1.0) / 12.0;
    return sigma / sqrt(var);
}

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    uint32_t lsb = (u >> 16) & 1u;
    u += 0x7FFFu + lsb;
    return (uint16_t)(u >> 16);
}

void synth_normal_f32(uint64_t seed, uint64_t tag, double mean, double sigma,
                      int64_t n, float *out) {
    uint64_t s0 = stream_base(seed, tag);
    double sc = ih8_scale(sigma);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) out[i] = (float)(mean + irwin_hall8(s0, (uint64_t)i, sc));
}

void synth_normal_bf16(uint64_t seed, uint64_t tag, double mean, double sigma,
                       int64_t n, uint16_t *out) {
    uint64_t s0 = stream_base(seed, tag);
    double sc = ih8_scale(sigma);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i)
        out[i] = f32_to_bf16_rne((float)(mean + irwin_hall8(s0, (uint64_t)i, sc)));
}

/* Uniform integers in [lo, lo + span) by the multiply-high map of the top 32
 * bits (bias below 2^-32 * span, irrelevant here).  span <= 2^32. */
void synth_uniform_i32(uint64_t seed, uint64_t tag, int64_t lo, int64_t span,
                       int64_t n, int32_t *out) {
    uint64_t s0 = stream_base(seed, tag);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i) {
        uint64_t r = raw_at(s0, (uint64_t)i) >> 32;
        out[i] = (int32_t)(lo + (int64_t)((r * (uint64_t)span) >> 32));
    }
}

/* Uniform doubles in [0, 1) with 53 random bits. */
void synth_uniform_f64(uint64_t seed, uint64_t tag, int64_t n, double *out) {
    uint64_t s0 = stream_base(seed, tag);
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < n; ++i)
        out[i] = (double)(raw_at(s0, (uint64_t)i) >> 11) * (1.0 / 9007199254740992.0);
}
