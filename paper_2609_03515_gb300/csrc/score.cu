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
constexpr int kScoreTok = 32;     // tokens per CTA (one per lane)

// CTA = 32 tokens x up to 32 layers.  Warp w computes s_l(i) of eligible layer
// k0 + w for the CTA's tokens (mean over the row's heads of exp2(z - lse2));
// warp 0 then folds the layers into the utility in ascending order.
__global__ void __launch_bounds__(kScoreWarps * 32) score_ema_kernel(const ScoreArgs a) {
    __shared__ float sl[kMaxLayersPerScorePass][kScoreTok];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.y;
    const int b = r / a.rows_per_seq;
    const int L = a.len[b];
    const int i0 = blockIdx.x * kScoreTok;
    if (i0 >= L) return;
    const int i = i0 + lane;
    const bool valid = i < L;
    int h0 = 0, nh = a.q_heads;
    if (a.rows_per_seq > 1) {
        nh = a.q_heads / a.kv_heads;
        h0 = (r % a.rows_per_seq) * nh;
    }
    const int H = a.q_heads;
    const float inv = 1.f / (float)nh;
    if (warp < a.n_elig) {
        const int li = a.elig[warp];
        const float *zl = a.logits + (((int64_t)b * a.n_layers + li) * H) * (int64_t)a.lstride;
        const float *ll = a.lse2 + ((int64_t)b * a.n_layers + li) * H;
        float acc = 0.f;
        if (valid) {
#pragma unroll 8
            for (int h = h0; h < h0 + nh; ++h) acc += exp2f(zl[(int64_t)h * a.lstride + i] - ll[h]);
        }
        sl[warp][lane] = acc * inv;
    }
    __syncthreads();
    if (warp == 0 && valid) {
        const int64_t at = (int64_t)r * a.cap + i;
        float m = a.ema ? a.ema[at] : 0.f;
        float sc = 0.f;
        for (int k = 0; k < a.n_elig; ++k) {
            sc = sl[k][lane];
            m = a.alpha * m + (1.f - a.alpha) * sc;
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

cudaError_t launch_score_ema(const ScoreArgs &a, int32_t max_len, cudaStream_t st) {
    if (max_len <= 0 || a.n_elig <= 0) return cudaSuccess;
    dim3 grid((max_len + kScoreTok - 1) / kScoreTok, a.batch * a.rows_per_seq);
    score_ema_kernel<<<grid, kScoreWarps * 32, 0, st>>>(a);
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
