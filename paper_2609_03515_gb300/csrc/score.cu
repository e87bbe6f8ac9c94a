// Eq. 1 score and the layer-sequential EMA of Eq. 4 (Appendix "Layer scoring"),
// fused with the softmax normalisation.
//
// score_ema_kernel: one CTA per (32-token chunk, utility row), one warp per
// eligible layer (up to 32 per pass), lanes over tokens.  Warp l computes
// s_l(i) = mean over the row's heads of p_h(i) = exp2(z_h(i) - lse2_h) from
// the attention kernel's log2-domain logits and log-sum-exp; warp 0 then folds
// the layers into the utility in ascending layer order,
// m = alpha m + (1 - alpha) s_l.  More than 32 eligible layers take several
// passes, launched in order.
#include "ikv_internal.cuh"

namespace ikv {
namespace {

constexpr int kScoreWarps = 32;   // one warp per eligible layer of a pass

template <int V> struct VecF;
template <> struct VecF<1> { using T = float; };
template <> struct VecF<2> { using T = float2; };
template <> struct VecF<4> { using T = float4; };
__device__ __forceinline__ float vget(float x, int) { return x; }
__device__ __forceinline__ float vget(float2 x, int v) { return v == 0 ? x.x : x.y; }
__device__ __forceinline__ float vget(float4 x, int v) { return v == 0 ? x.x : v == 1 ? x.y : v == 2 ? x.z : x.w; }

// CTA = 32 V tokens x up to 32 layers.  Warp w computes s_l(i) of eligible
// layer k0 + w for the CTA's tokens (mean over the row's heads of
// exp2(z - lse2)), V consecutive tokens per lane; the CTA's first 32 V
// threads then fold the layers into the utility in ascending order.  The
// pass is latency bound: every head of a batch of 32 / V is loaded before any
// is used, the per-head log-sum-exp travels by shuffle, and the utility is
// fetched before the loads.  V > 1 reads each head row in 256- or 512-byte
// runs, which DRAM serves far better than scattered 128-byte pieces.
template <int V>
__global__ void __launch_bounds__(kScoreWarps * 32, 1) score_ema_kernel(const ScoreArgs a) {
    using VT = typename VecF<V>::T;
    constexpr int kTok = 32 * V;   // tokens per CTA
    constexpr int kHB = 32 / V;    // heads per load batch (32 registers of loads)
    __shared__ __align__(16) float sl[kMaxLayersPerScorePass][kTok];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.y;
    const int b = r / a.rows_per_seq;
    const int L = a.len[b];
    const int i0 = blockIdx.x * kTok;
    if (i0 >= L) return;
    const int il = i0 + lane * V;  // first token of this lane
    int h0 = 0, nh = a.q_heads;
    if (a.rows_per_seq > 1) {
        nh = a.q_heads / a.kv_heads;
        h0 = (r % a.rows_per_seq) * nh;
    }
    const int H = a.q_heads;
    const float inv = 1.f / (float)nh;
    const int fi = i0 + (int)threadIdx.x;  // token folded by this thread (threads < kTok)
    const bool folds = threadIdx.x < kTok && fi < L;
    const int64_t at = (int64_t)r * a.cap + fi;
    float m = 0.f;
    if (folds && a.ema) m = a.ema[at];
    if (warp < a.n_elig) {
        const int li = a.elig[warp];
        // row padding keeps i0 + kTok <= lstride, so the vector loads stay inside the row
        const float *zp = a.logits + (((int64_t)b * a.n_layers + li) * H + h0) * (int64_t)a.lstride + il;
        const float *ll = a.lse2 + ((int64_t)b * a.n_layers + li) * H + h0;
        float acc[V];
#pragma unroll
        for (int v = 0; v < V; ++v) acc[v] = 0.f;
        for (int hb = 0; hb < nh; hb += kHB) {
            const int nb = min(kHB, nh - hb);
            const float lse_lane = lane < nb ? ll[hb + lane] : 0.f;
            VT z[kHB];
#pragma unroll
            for (int j = 0; j < kHB; ++j) {
                if (il < L && j < nb) z[j] = __ldg(reinterpret_cast<const VT *>(zp));
                zp += a.lstride;
            }
#pragma unroll
            for (int j = 0; j < kHB; ++j) {
                const float lj = __shfl_sync(0xffffffffu, lse_lane, j);
                if (il < L && j < nb) {
#pragma unroll
                    for (int v = 0; v < V; ++v) acc[v] += exp2f(vget(z[j], v) - lj);
                }
            }
        }
#pragma unroll
        for (int v = 0; v < V; ++v) sl[warp][lane * V + v] = acc[v] * inv;
    }
    __syncthreads();
    if (folds) {
        float sc = 0.f;
        for (int k = 0; k < a.n_elig; ++k) {
            sc = sl[k][threadIdx.x];
            if (a.agg == IKV_AGG_EMA)
                m = a.alpha * m + (1.f - a.alpha) * sc;  // Eq. 4
            else if (a.agg == IKV_AGG_CUMULATIVE)
                m += sc;                                  // Eq. 3
            else
                m = sc;                                   // Eq. 2
        }
        if (a.ema) a.ema[at] = m;
        if (a.score) a.score[at] = sc;
    }
}

__global__ void ema_update_kernel(int32_t cap, float *ema, const float *score, const int32_t *len, int32_t rps,
                                  float alpha) {
    const int r = blockIdx.y;
    const int L = len[r / rps];
    for (int i = blockIdx.x * blockDim.x + threadIdx.x; i < L; i += gridDim.x * blockDim.x) {
        const int64_t at = (int64_t)r * cap + i;
        ema[at] = alpha * ema[at] + (1.f - alpha) * score[at];
    }
}

}  // namespace

cudaError_t launch_score_ema(const ScoreArgs &a, int32_t max_len, int sms, cudaStream_t st) {
    if (max_len <= 0 || a.n_elig <= 0) return cudaSuccess;
    // widest token vector that still gives every SM two CTAs
    const int64_t rows = (int64_t)a.batch * a.rows_per_seq;
    auto ctas = [&](int tok) { return rows * ((max_len + tok - 1) / tok); };
    const int V = ctas(128) >= 2 * sms ? 4 : ctas(64) >= 2 * sms ? 2 : 1;
    dim3 grid((max_len + 32 * V - 1) / (32 * V), (unsigned)rows);
    if (V == 4)
        score_ema_kernel<4><<<grid, kScoreWarps * 32, 0, st>>>(a);
    else if (V == 2)
        score_ema_kernel<2><<<grid, kScoreWarps * 32, 0, st>>>(a);
    else
        score_ema_kernel<1><<<grid, kScoreWarps * 32, 0, st>>>(a);
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_ema_update(int32_t rows, int32_t cap, float *ema, const float *score, const int32_t *len,
                              int32_t rows_per_seq, float alpha, int32_t max_len, cudaStream_t st) {
    if (rows <= 0 || max_len <= 0) return cudaSuccess;
    int gx = (max_len + 255) / 256;
    if (gx > 1024) gx = 1024;
    ema_update_kernel<<<dim3(gx, rows), 256, 0, st>>>(cap, ema, score, len, rows_per_seq, alpha);
    note_launch();
    return cudaGetLastError();
}

}  // namespace ikv
