/*
 * Host side of the synthetic workload generator (see ikvgen.h for the recipe).
 * Compiled with gcc -O2 -fopenmp -ffp-contract=off; used by the CPU oracle
 * tests and by the benchmark's CPU baseline to reproduce the exact inputs the
 * device generator wrote.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#include "ikvgen.h"

static void store(void *out, int64_t idx, float v, int dtype) {
    if (dtype == IKVGEN_BF16)
        ((uint16_t *)out)[idx] = ikvgen_bf16_bits(v);
    else
        ((float *)out)[idx] = v;
}

/* u(l,g,:) = sqrt(d) * n / |n|, n ~ N(0,I); computed in fp64, stored fp32. */
void ikvgen_u_table(uint64_t seed, int32_t layers, int32_t kv_heads, int32_t d, float *out) {
    for (int32_t l = 0; l < layers; ++l)
        for (int32_t g = 0; g < kv_heads; ++g) {
            double nrm = 0.0;
            double tmp[1024];
            for (int32_t e = 0; e < d; ++e) {
                tmp[e] = (double)ikvgen_normal(seed, IKVGEN_S_UDIR, (uint64_t)l, ikvgen_w1(0, g, e));
                nrm += tmp[e] * tmp[e];
            }
            double sc = sqrt((double)d) / sqrt(nrm);
            for (int32_t e = 0; e < d; ++e) out[((int64_t)l * kv_heads + g) * d + e] = (float)(tmp[e] * sc);
        }
}

/* Keys and values of sequence b, layer l, positions [p0, p0+count), all kv heads.
 * out_k / out_v: [kv_heads][count][d] (either may be NULL). */
void ikvgen_kv_block(const ikvgen_spec *s, const float *u, int32_t b, int32_t l, int64_t p0, int64_t count,
                     int32_t dtype, void *out_k, void *out_v) {
    const int32_t d = s->head_dim;
#pragma omp parallel for schedule(static) collapse(2)
    for (int32_t g = 0; g < s->kv_heads; ++g)
        for (int64_t i = 0; i < count; ++i) {
            int64_t p = p0 + i;
            int heavy = ikvgen_is_heavy(s, b, p);
            const float *ug = u + ((int64_t)l * s->kv_heads + g) * d;
            int64_t base = ((int64_t)g * count + i) * d;
            for (int32_t e = 0; e < d; ++e) {
                if (out_k) store(out_k, base + e, ikvgen_key_elem(s, b, l, g, p, e, heavy, ug[e]), dtype);
                if (out_v) store(out_v, base + e, ikvgen_value_elem(s, b, l, g, p, e), dtype);
            }
        }
}

/* Keys and values of sequence b, layer l at the listed positions (any order).
 * out_k / out_v: [kv_heads][count][d] (either may be NULL). */
void ikvgen_kv_rows_at(const ikvgen_spec *s, const float *u, int32_t b, int32_t l, const int64_t *positions,
                       int64_t count, int32_t dtype, void *out_k, void *out_v) {
    const int32_t d = s->head_dim;
#pragma omp parallel for schedule(static) collapse(2)
    for (int32_t g = 0; g < s->kv_heads; ++g)
        for (int64_t i = 0; i < count; ++i) {
            int64_t p = positions[i];
            int heavy = ikvgen_is_heavy(s, b, p);
            const float *ug = u + ((int64_t)l * s->kv_heads + g) * d;
            int64_t base = ((int64_t)g * count + i) * d;
            for (int32_t e = 0; e < d; ++e) {
                if (out_k) store(out_k, base + e, ikvgen_key_elem(s, b, l, g, p, e, heavy, ug[e]), dtype);
                if (out_v) store(out_v, base + e, ikvgen_value_elem(s, b, l, g, p, e), dtype);
            }
        }
}

/* Heavy-position flags for positions [p0, p0+count) of sequence b. */
void ikvgen_heavy_flags(const ikvgen_spec *s, int32_t b, int64_t p0, int64_t count, uint8_t *out) {
    for (int64_t i = 0; i < count; ++i) out[i] = (uint8_t)ikvgen_is_heavy(s, b, p0 + i);
}

/* Queries for decode steps t in [t0, t1) (1-based):
 * out [t1-t0][layers][batch][q_heads][d].  mode 0: w_t = 0.5*eps_t; mode 1: w_t = w_{t-1} + 0.1*eps_t. */
void ikvgen_queries(uint64_t seed, int32_t batch, int32_t layers, int32_t q_heads, int32_t kv_heads, int32_t d,
                    const float *u, int32_t mode, int32_t t0, int32_t t1, int32_t dtype, void *out) {
    const int32_t grp = q_heads / kv_heads;
    const int64_t per_step = (int64_t)layers * batch * q_heads * d;
#pragma omp parallel for schedule(static) collapse(3)
    for (int32_t l = 0; l < layers; ++l)
        for (int32_t b = 0; b < batch; ++b)
            for (int32_t h = 0; h < q_heads; ++h) {
                double w[1024];
                double x[1024];
                const float *ug = u + ((int64_t)l * kv_heads + h / grp) * d;
                for (int32_t e = 0; e < d; ++e) w[e] = 0.0;
                for (int32_t t = (mode == 1 ? 1 : t0); t < t1; ++t) {
                    for (int32_t e = 0; e < d; ++e) {
                        double eps = (double)ikvgen_normal(seed, IKVGEN_S_QUERY, ikvgen_w0(b, t), ikvgen_w1(l, h, e));
                        w[e] = (mode == 1) ? w[e] + 0.1 * eps : 0.5 * eps;
                    }
                    if (t < t0) continue;
                    double nrm = 0.0;
                    for (int32_t e = 0; e < d; ++e) {
                        x[e] = (double)ug[e] + w[e];
                        nrm += x[e] * x[e];
                    }
                    double sc = sqrt((double)d) / sqrt(nrm);
                    int64_t base = (int64_t)(t - t0) * per_step + (((int64_t)l * batch + b) * q_heads + h) * d;
                    for (int32_t e = 0; e < d; ++e) store(out, base + e, (float)(x[e] * sc), dtype);
                }
            }
}

/* Per-sequence prefill lengths, uniform integers in [lo, hi]. */
void ikvgen_lengths(uint64_t seed, int32_t batch, int32_t lo, int32_t hi, int32_t *out) {
    for (int32_t b = 0; b < batch; ++b) {
        uint64_t h = ikvgen_hash(seed, IKVGEN_S_LEN, (uint64_t)b, 0);
        out[b] = lo + (int32_t)(h % (uint64_t)(hi - lo + 1));
    }
}

/* Raw draws, exported so tests can check the distribution and host/device agreement. */
void ikvgen_normals(uint64_t seed, uint64_t stream, int64_t n, float *out) {
    for (int64_t i = 0; i < n; ++i) out[i] = ikvgen_normal(seed, stream, (uint64_t)i, 0);
}

uint64_t ikvgen_mix64_host(uint64_t z) { return ikvgen_mix64(z); }
