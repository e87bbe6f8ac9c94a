// Eq. 1 score and the layer-sequential EMA of Eq. 4 (Appendix "Layer scoring"),
// fused with the softmax normalisation.
//
// score_ema_kernel: one CTA per (32-token chunk, utility row).  Lanes own
// tokens; the 8 warps split the row's query heads.  For every eligible layer a
// warp sums p_h(i) = exp2(z_h(i) - lse2_h) over its heads (the attention
// kernel's log2-domain logits, normalised by the combine's log-sum-exp); the
// per-warp partials meet in shared memory, and warp 0 folds the layers into
// the utility in ascending layer order: m = alpha m + (1 - alpha) s_l.
#include "ikv_internal.cuh"

namespace ikv {
namespace {

constexpr int kScoreWarps = 8;

__global__ void __launch_bounds__(kScoreWarps * 32) score_ema_kernel(const ScoreArgs a) {
    __shared__ float red[kMaxLayersPerScorePass][kScoreWarps][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.y;
    const int b = r / a.rows_per_seq;
    const int L = a.len[b];
    const int i0 = blockIdx.x * 32;
    if (i0 >= L) return;
    const int i = i0 + lane;
    const bool valid = i < L;
    int h0 = 0, nh = a.q_heads;
    if (a.rows_per_seq > 1) {
        nh = a.q_heads / a.kv_heads;
        h0 = (r % a.rows_per_seq) * nh;
    }
    const int H = a.q_heads;
    for (int k = 0; k < a.n_elig; ++k) {
        const int li = a.elig[k];
        const float *zl = a.logits + (((int64_t)b * a.n_layers + li) * H) * (int64_t)a.cap;
        const float *ll = a.lse2 + ((int64_t)b * a.n_layers + li) * H;
        float acc = 0.f;
        if (valid) {
#pragma unroll 4
            for (int h = h0 + warp; h < h0 + nh; h += kScoreWarps) acc += exp2f(zl[(int64_t)h * a.cap + i] - ll[h]);
        }
        red[k][warp][lane] = acc;
    }
    __syncthreads();
    if (warp == 0 && valid) {
        const int64_t at = (int64_t)r * a.cap + i;
        float m = a.ema ? a.ema[at] : 0.f;
        const float inv = 1.f / (float)nh;
        float sc = 0.f;
        for (int k = 0; k < a.n_elig; ++k) {
            float s = 0.f;
#pragma unroll
            for (int w = 0; w < kScoreWarps; ++w) s += red[k][w][lane];
            sc = s * inv;
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
    dim3 grid((max_len + 31) / 32, a.batch * a.rows_per_seq);
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
