// Per-layer immediate eviction (IKV_EVICT_LAYER): every layer folds its Eq. 1 score
// into a state indexed by token position and shared by all layers, then keeps the
// budget's highest-utility tokens among those it holds (Appendix "Layer scoring",
// each layer's hook acting at once).  A live position that a layer does not hold gets
// score 0 there, so Eq. 4 multiplies it by alpha; rather than touching every live
// position at every layer, the decay is applied when the position is next read (its
// pending count is the eligible layers since its last update) and, for the rest, once
// at the end of the step.
#include "ikv_internal.cuh"

namespace ikv {

__device__ unsigned int g_layer_error = 0;  // bit 2: no free slot; bit 3: next_pos reached pos_cap

namespace {

constexpr int kBeginThreads = 1024;

// alpha^n by repeated multiplication, n >= 0 (at most the layer count)
__device__ __forceinline__ float decay(float v, float alpha, int n) {
    for (int i = 0; i < n; ++i) v *= alpha;
    return v;
}

// One CTA per sequence: the new token's state (0, or the mean over the positions some
// layer holds, found by marking them in lam), its position in every layer's row, the
// pending-update marks reset, then len and next_pos advanced.
__global__ void __launch_bounds__(kBeginThreads) layer_begin_kernel(const LayerArgs a) {
    pdl_wait();
    __shared__ float red[2][kBeginThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.x;
    const int L = a.len[b];
    const int S = a.start ? a.start[b] : 0;
    const int np = a.next_pos[b];
    int32_t *lam = a.lam + (int64_t)b * a.pos_cap;
    float *m = a.m + (int64_t)b * a.pos_cap;
    if (S + L >= a.cap || np >= a.pos_cap) {
        if (tid == 0) {
            a.slot[b] = -1;
            atomicOr(&g_layer_error, S + L >= a.cap ? 4u : 8u);
        }
        return;
    }
    float init = 0.f;
    if (a.init_mean) {
        for (int p = tid; p < np; p += kBeginThreads) lam[p] = 0;
        __syncthreads();
        for (int64_t i = tid; i < (int64_t)a.layers * L; i += kBeginThreads) {
            const int l = (int)(i / L), j = (int)(i % L);
            const int p = a.pos[((int64_t)b * a.layers + l) * a.cap + j];
            if (p >= 0 && p < np) lam[p] = 1;
        }
        __syncthreads();
        float sum = 0.f, cnt = 0.f;
        for (int p = tid; p < np; p += kBeginThreads)
            if (lam[p] == 1) {
                sum += m[p];
                cnt += 1.f;
            }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            sum += __shfl_xor_sync(0xffffffffu, sum, o);
            cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
        }
        if (lane == 0) red[0][warp] = sum, red[1][warp] = cnt;
        __syncthreads();
        float ts = 0.f, tc = 0.f;
        for (int w = 0; w < kBeginThreads / 32; ++w) ts += red[0][w], tc += red[1][w];
        init = tc > 0.f ? ts / tc : 0.f;
    }
    __syncthreads();  // every thread has read len / next_pos and the marks
    for (int p = tid; p <= np; p += kBeginThreads) lam[p] = -1;
    for (int l = tid; l < a.layers; l += kBeginThreads) a.pos[((int64_t)b * a.layers + l) * a.cap + L] = np;
    if (tid == 0) {
        m[np] = init;
        a.slot[b] = L;
        a.next_pos[b] = np + 1;
        a.len[b] = L + 1;
    }
}

// One thread per slot j of layer `layer`: the position's utility as of this layer
// (pending decays applied), with this layer's Eq. 1 score folded in on scoring layers
// (then stored back, marked as updated by this layer).  Writes util[b][j].
constexpr int kUtilThreads = 256;
__global__ void __launch_bounds__(kUtilThreads) layer_util_kernel(const LayerArgs a) {
    pdl_wait();
    const int b = blockIdx.y;
    const int j = blockIdx.x * kUtilThreads + threadIdx.x;
    const int L = a.len[b];
    if (j >= L) return;
    const int p = a.pos[((int64_t)b * a.layers + a.layer) * a.cap + j];
    float *util = a.util + (int64_t)b * a.cap;
    if (p < 0 || p >= a.pos_cap) {  // not a valid position: never kept
        util[j] = -INFINITY;
        return;
    }
    float *m = a.m + (int64_t)b * a.pos_cap;
    int32_t *lam = a.lam + (int64_t)b * a.pos_cap;
    float v = decay(m[p], a.alpha, (a.k_done - 1) - lam[p]);
    if (a.scoring) {
        const int H = a.q_heads;
        const int64_t row = (int64_t)b * a.sc_layers + a.layer;
        const float *z = a.logits + row * H * (int64_t)a.lstride + j;
        const float *l2 = a.lse2 + row * H;
        float s = 0.f;
        for (int h = 0; h < H; ++h) s += exp2f(__ldg(z + (int64_t)h * a.lstride) - __ldg(l2 + h));
        v = a.alpha * v + (1.f - a.alpha) * (s / (float)H);
        m[p] = v;
        lam[p] = a.k_done;
    }
    util[j] = v;
}

// End of a step: the decays still pending (eligible layers after a position's last
// update) are applied to every position below next_pos; len becomes the kept count.
constexpr int kEndThreads = 256;
__global__ void __launch_bounds__(kEndThreads) layer_end_kernel(const LayerArgs a) {
    pdl_wait();
    const int b = blockIdx.y;
    const int p = blockIdx.x * kEndThreads + threadIdx.x;
    if (a.n_elig > 0 && p < a.next_pos[b] && p < a.pos_cap) {
        float *m = a.m + (int64_t)b * a.pos_cap;
        const int32_t *lam = a.lam + (int64_t)b * a.pos_cap;
        m[p] = decay(m[p], a.alpha, (a.n_elig - 1) - lam[p]);
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) a.len[b] = a.keep_len[b];
}

}  // namespace

cudaError_t launch_layer_begin(const LayerArgs &a, cudaStream_t st) {
    cudaError_t e = launch_k(layer_begin_kernel, dim3(a.batch), dim3(kBeginThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_layer_util(const LayerArgs &a, int32_t max_len, cudaStream_t st) {
    if (max_len <= 0) return cudaSuccess;
    dim3 grid((max_len + kUtilThreads - 1) / kUtilThreads, a.batch);
    cudaError_t e = launch_k(layer_util_kernel, grid, dim3(kUtilThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_layer_end(const LayerArgs &a, cudaStream_t st) {
    dim3 grid((a.pos_cap + kEndThreads - 1) / kEndThreads, a.batch);
    cudaError_t e = launch_k(layer_end_kernel, grid, dim3(kEndThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t read_clear_layer_error(unsigned int *v) {
    unsigned int z = 0;
    cudaError_t e = cudaMemcpyFromSymbol(v, g_layer_error, sizeof(*v));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_layer_error, &z, sizeof(z));
    return e;
}

}  // namespace ikv
