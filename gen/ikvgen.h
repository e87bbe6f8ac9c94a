/*
 * ikvgen.h -- seeded synthetic decode workload generator (inputs only).
 *
 * This module produces the keys, values and queries that both the CUDA path
 * and the CPU oracle consume.  It holds none of the eviction method's
 * arithmetic: it only draws numbers.  The same element functions are compiled
 * for the host (gcc, libikvgen_host.so) and for the device (nvcc,
 * libikvgen_cuda.so) so that a prefilled cache written on the GPU can be
 * reproduced row by row on the CPU, bit for bit.
 *
 * Bit-reproducibility rules followed below:
 *   - integers only up to the final int->float conversion of a normal draw;
 *   - every later float operation is a single IEEE round-to-nearest op
 *     (device: __fmul_rn/__fadd_rn, host: plain float ops compiled with
 *     -ffp-contract=off so no FMA contraction happens on aarch64 either);
 *   - bf16 is produced by round-to-nearest-even on the fp32 bits.
 *
 * Generator: the SplitMix64 output function (Steele, Lea, Flood, "Fast
 * splittable pseudorandom number generators", OOPSLA 2014, with the mixing
 * constants published by Vigna), used as a counter-based hash.
 * Normal draws: Irwin-Hall with twelve 16-bit uniforms, centred, which has
 * mean 0 and variance 1 (up to 2^-32) and is exact in fp32.
 *
 * Workload recipe (synthetic stand-in for the paper's long-context runs):
 *   key  k(b,l,g,p,:) = N(0,I)                          ordinary token
 *                     = 3*u(l,g,:) + 0.3*N(0,I)         heavy token (1% of positions per sequence)
 *                       then x sink_scale for positions p < n_sinks
 *   value v(b,l,g,p,:) = N(0,I)
 *   u(l,g,:) : fixed direction per (layer, kv head) with norm sqrt(d)
 *   query q_t(b,l,h,:) = sqrt(d) * normalize(u(l,g(h),:) + w_t(b,l,h,:)),
 *       w_t = 0.5*eps_t (iid mode)  or  w_t = w_{t-1} + 0.1*eps_t, w_0 = 0 (walk mode)
 */
#ifndef IKVGEN_H
#define IKVGEN_H

#include <stdint.h>

#if defined(__CUDACC__)
#define IKVGEN_HD __host__ __device__ __forceinline__
#else
#define IKVGEN_HD static inline
#endif

/* streams: keep the draws of different tensors independent */
#define IKVGEN_S_KEY    1ull
#define IKVGEN_S_VALUE  2ull
#define IKVGEN_S_HEAVY  3ull
#define IKVGEN_S_QUERY  4ull
#define IKVGEN_S_UDIR   5ull
#define IKVGEN_S_LEN    6ull

#define IKVGEN_F32  0
#define IKVGEN_BF16 1

typedef struct {
    uint64_t seed;
    int32_t batch, layers, kv_heads, head_dim;
    int32_t heavy_per_10000;   /* 100 -> 1% heavy positions */
    int32_t n_sinks;           /* first positions whose keys are scaled */
    float sink_scale;          /* 4.0 */
    float heavy_u_scale;       /* 3.0 */
    float heavy_noise;         /* 0.3 */
} ikvgen_spec;

IKVGEN_HD uint64_t ikvgen_mix64(uint64_t z) {
    z += 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

IKVGEN_HD uint64_t ikvgen_hash(uint64_t seed, uint64_t stream, uint64_t w0, uint64_t w1) {
    uint64_t x = ikvgen_mix64(seed ^ (stream * 0xD1B54A32D192ED03ull));
    x = ikvgen_mix64(x ^ w0);
    return ikvgen_mix64(x ^ w1);
}

/* Irwin-Hall(12) normal from a 64-bit counter state; exact in fp32. */
IKVGEN_HD float ikvgen_normal_from(uint64_t h) {
    int64_t s = 0;
    for (int r = 0; r < 3; ++r) {
        uint64_t z = ikvgen_mix64(h + (uint64_t)r);
        s += (int64_t)(z & 0xFFFF) + (int64_t)((z >> 16) & 0xFFFF) +
             (int64_t)((z >> 32) & 0xFFFF) + (int64_t)(z >> 48);
    }
    /* sum of 12 uniforms on {0..65535}; E = 12*32767.5 = 393210 */
    return (float)(s - 393210) * (1.0f / 65536.0f);
}

IKVGEN_HD float ikvgen_normal(uint64_t seed, uint64_t stream, uint64_t w0, uint64_t w1) {
    return ikvgen_normal_from(ikvgen_hash(seed, stream, w0, w1));
}

IKVGEN_HD int ikvgen_is_heavy(const ikvgen_spec *s, int32_t b, int64_t p) {
    uint64_t h = ikvgen_hash(s->seed, IKVGEN_S_HEAVY, (uint64_t)b, (uint64_t)p);
    return (int)(h % 10000ull) < s->heavy_per_10000;
}

IKVGEN_HD uint64_t ikvgen_w0(int32_t b, int64_t p) { return ((uint64_t)(uint32_t)b << 40) ^ (uint64_t)p; }
IKVGEN_HD uint64_t ikvgen_w1(int32_t l, int32_t g, int32_t e) {
    return ((uint64_t)(uint32_t)l << 32) ^ ((uint64_t)(uint32_t)g << 16) ^ (uint64_t)(uint32_t)e;
}

IKVGEN_HD float ikvgen_mul(float a, float b) {
#if defined(__CUDA_ARCH__)
    return __fmul_rn(a, b);
#else
    return a * b;
#endif
}
IKVGEN_HD float ikvgen_add(float a, float b) {
#if defined(__CUDA_ARCH__)
    return __fadd_rn(a, b);
#else
    return a + b;
#endif
}

/* key element; heavy_flag and u_e are passed in so a row costs one flag draw */
IKVGEN_HD float ikvgen_key_elem(const ikvgen_spec *s, int32_t b, int32_t l, int32_t g, int64_t p,
                                int32_t e, int heavy_flag, float u_e) {
    float n = ikvgen_normal(s->seed, IKVGEN_S_KEY, ikvgen_w0(b, p), ikvgen_w1(l, g, e));
    float k = n;
    if (heavy_flag) k = ikvgen_add(ikvgen_mul(s->heavy_u_scale, u_e), ikvgen_mul(s->heavy_noise, n));
    if (p < s->n_sinks) k = ikvgen_mul(s->sink_scale, k);
    return k;
}

IKVGEN_HD float ikvgen_value_elem(const ikvgen_spec *s, int32_t b, int32_t l, int32_t g, int64_t p,
                                  int32_t e) {
    return ikvgen_normal(s->seed, IKVGEN_S_VALUE, ikvgen_w0(b, p), ikvgen_w1(l, g, e));
}

/* fp32 -> bf16 bits, round to nearest even (inputs here are always finite) */
IKVGEN_HD uint16_t ikvgen_bf16_bits(float f) {
    union { float f; uint32_t u; } c;
    c.f = f;
    uint32_t x = c.u;
    x += 0x7FFFu + ((x >> 16) & 1u);
    return (uint16_t)(x >> 16);
}

#endif /* IKVGEN_H */
