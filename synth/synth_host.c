/*
 * synth_host.c - seeded synthetic inputs (host side).
 *
 * This module generates the inputs that both the CUDA decode path and the
 * fp64 oracle consume: random-init bf16 weights and uniform prompt tokens.
 * It holds none of the decoding method's arithmetic.  The device twin in
 * synth_dev.cu implements the same definition; a test checks the two agree
 * bit for bit.
 *
 * Definition of weight element i of tensor t under seed s:
 *   key  = (t << 40) | i                              (i < 2^40)
 *   s'   = mix64(s + 0x9E3779B97F4A7C15)
 *   w0   = mix64(s' ^ (2*key)),  w1 = mix64(s' ^ (2*key + 1))
 *   S    = sum of the eight 16-bit fields of w0 and w1   (0 <= S <= 8*65535)
 *   v    = (double)(S - 262140) * c                      (one IEEE multiply)
 *   out  = bf16_rne(float_rne(v))
 * mix64 is the SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014,
 * with Stafford's "Mix13" constants).  S is an Irwin-Hall(8) variable with
 * mean 262140 and standard deviation 53509.92; the caller passes
 * c = sigma * scale / 53509.92 so v approximates N(0, (sigma*scale)^2).
 * Rounding double -> float -> bf16 (both round-to-nearest-even) is the same
 * two-step rounding torch applies in tensor(fp64).to(bfloat16).
 *
 * Prompt token i under seed s: mix64(s' ^ ((0xFFFFull << 40) | i)) % vocab.
 */
#include <stdint.h>
#include <string.h>

static inline uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static inline uint16_t f32_to_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

static inline int64_t irwin_hall8(uint64_t s2, uint64_t key) {
    uint64_t w0 = mix64(s2 ^ (2u * key));
    uint64_t w1 = mix64(s2 ^ (2u * key + 1u));
    int64_t s = 0;
    for (int b = 0; b < 4; ++b) {
        s += (int64_t)((w0 >> (16 * b)) & 0xFFFFu);
        s += (int64_t)((w1 >> (16 * b)) & 0xFFFFu);
    }
    return s - 262140;
}

/* Fill out[0..n) with bf16 bits of tensor `tensor_id`, elements
 * [first, first+n) of its flat index space. */
void synth_fill_bf16(uint16_t* out, uint64_t first, uint64_t n, uint64_t seed,
                     uint32_t tensor_id, double c) {
    const uint64_t s2 = mix64(seed + 0x9E3779B97F4A7C15ull);
    const uint64_t base = ((uint64_t)tensor_id) << 40;
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < (int64_t)n; ++j) {
        uint64_t key = base | (first + (uint64_t)j);
        double v = (double)irwin_hall8(s2, key) * c;
        out[j] = f32_to_bf16_rne((float)v);
    }
}

/* Same generator, widened: fp64 values before any rounding (used to fill the
 * oracle's fp64 KV cache for timing runs at a given context length). */
void synth_fill_f64(double* out, uint64_t first, uint64_t n, uint64_t seed,
                    uint32_t tensor_id, double c) {
    const uint64_t s2 = mix64(seed + 0x9E3779B97F4A7C15ull);
    const uint64_t base = ((uint64_t)tensor_id) << 40;
    #pragma omp parallel for schedule(static)
    for (int64_t j = 0; j < (int64_t)n; ++j) {
        uint64_t key = base | (first + (uint64_t)j);
        out[j] = (double)irwin_hall8(s2, key) * c;
    }
}

/* Uniform prompt tokens over [0, vocab). */
void synth_prompt(int32_t* out, int n, uint64_t seed, int vocab) {
    const uint64_t s2 = mix64(seed + 0x9E3779B97F4A7C15ull);
    for (int i = 0; i < n; ++i) {
        uint64_t key = (0xFFFFull << 40) | (uint64_t)i;
        out[i] = (int32_t)(mix64(s2 ^ key) % (uint64_t)vocab);
    }
}

/* Bare rounding helper exposed for the rounding test against torch. */
void synth_round_bf16(const double* in, uint16_t* out, uint64_t n) {
    for (uint64_t j = 0; j < n; ++j) out[j] = f32_to_bf16_rne((float)in[j]);
}
