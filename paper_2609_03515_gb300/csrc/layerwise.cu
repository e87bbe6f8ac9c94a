// Per-layer immediate eviction (IKV_EVICT_LAYER): every layer folds its Eq. 1 score
// into a state indexed by token position and shared by all layers, then keeps the
// budget's highest-utility tokens among those it holds (Appendix "Layer scoring",
// each layer's hook acting at once).  A live position that a layer does not hold gets
// score 0 there, so Eq. 4 multiplies it by alpha.
//
// No layer's eviction changes another layer's inputs within a step: a layer attends
// its own rows, and its update reads only the tokens it held before the step's
// evictions.  So after all attention (and the stored per-layer scores), one pass over
// token positions walks the layers in order -- the state as each layer saw it is that
// layer's utility for its slot of the position -- and every layer is then selected
// and compacted at once by the step's usual kernels (rows = batch x layers).
#include "ikv_internal.cuh"

namespace ikv {

__device__ unsigned int g_layer_error = 0;  // bit 2: no free slot; bit 3: next_pos reached pos_cap

namespace {

constexpr int kBeginThreads = 1024;

// The live positions (held by some layer) as bits, set by one thread per (sequence,
// layer, slot) into the cleared bitmap.  Nothing is evicted between here and the fold,
// so with the new token's bit (set by the begin kernel) this is the fold's live set.
constexpr int kMarkThreads = 256;
__global__ void __launch_bounds__(kMarkThreads) layer_mark_kernel(const LayerArgs a) {
    pdl_wait();
    const int b = blockIdx.z, l = blockIdx.y;
    const int j = blockIdx.x * kMarkThreads + threadIdx.x;
    if (j >= a.len[b]) return;
    const int p = a.pos[((int64_t)b * a.layers + l) * a.cap + j];
    if (p >= 0 && p < a.pos_cap) atomicOr(a.live + (int64_t)b * a.live_words + (p >> 5), 1u << (p & 31));
}

// One CTA per sequence: the new token's state (0, or the mean over the live positions),
// its live bit and position in every layer's row, then len and next_pos advanced.
__global__ void __launch_bounds__(kBeginThreads) layer_begin_kernel(const LayerArgs a) {
    pdl_wait();
    __shared__ float red[2][kBeginThreads / 32];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int b = blockIdx.x;
    const int L = a.len[b];
    const int S = a.start ? a.start[b] : 0;
    const int np = a.next_pos[b];
    float *m = a.m + (int64_t)b * a.pos_cap;
    uint32_t *bits = a.live + (int64_t)b * a.live_words;
    if (S + L >= a.cap || np >= a.pos_cap) {
        if (tid == 0) {
            a.slot[b] = -1;
            atomicOr(&g_layer_error, S + L >= a.cap ? 4u : 8u);
        }
        return;
    }
    float init = 0.f;
    if (a.init_mean) {
        float sum = 0.f, cnt = 0.f;
        for (int p = tid; p < np; p += kBeginThreads)
            if ((bits[p >> 5] >> (p & 31)) & 1u) {
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
    __syncthreads();  // every thread has read len / next_pos and the bits
    for (int l = tid; l < a.layers; l += kBeginThreads) a.pos[((int64_t)b * a.layers + l) * a.cap + L] = np;
    if (tid == 0) {
        bits[np >> 5] |= 1u << (np & 31);  // the new token is live too
        m[np] = init;
        a.slot[b] = L;
        a.next_pos[b] = np + 1;
        a.len[b] = L + 1;
    }
}

// inv[b][l][pos[b][l][j]] = j for every slot j < len[b] of every layer
constexpr int kInvThreads = 256;
__global__ void __launch_bounds__(kInvThreads) layer_inverse_kernel(const LayerArgs a) {
    pdl_wait();
    const int b = blockIdx.z, l = blockIdx.y;
    const int j = blockIdx.x * kInvThreads + threadIdx.x;
    if (j >= a.len[b]) return;
    const int p = a.pos[((int64_t)b * a.layers + l) * a.cap + j];
    if (p >= 0 && p < a.pos_cap) a.inv[((int64_t)b * a.layers + l) * a.pos_cap + p] = j;
}

// One thread per live token position p (held by some layer): walks the layers in
// order; at every eligible layer of a refresh step m <- alpha m + (1 - alpha) s, s the
// layer's pooled score of p if it holds p, else 0; each layer holding p gets m as its
// utility of p's slot.  The final m is stored.  Dead positions are left as they are.
constexpr int kFoldThreads = 256;
// 8, 16 and 32 measured alike (~15 us per fold at 32 layers x 3.3k slots): past the first
// batch the fold is bound by its scattered reads, not by their latency chain
#ifndef IKV_FOLD_BATCH
#define IKV_FOLD_BATCH 8
#endif
constexpr int kFoldBatch = IKV_FOLD_BATCH;  // layers whose lookups are in flight together
__global__ void __launch_bounds__(kFoldThreads) layer_fold_kernel(const LayerArgs a) {
    pdl_wait();
    const int b = blockIdx.y;
    const int p = blockIdx.x * kFoldThreads + threadIdx.x;
    if (p >= a.next_pos[b] || p >= a.pos_cap) return;
    if (!((__ldg(a.live + (int64_t)b * a.live_words + (p >> 5)) >> (p & 31)) & 1u)) return;
    const int L = a.len[b];
    float *mp = a.m + (int64_t)b * a.pos_cap + p;
    float m = *mp;
    int k = 0;  // eligible layers folded so far
    for (int l0 = 0; l0 < a.layers; l0 += kFoldBatch) {
        // the batch's slot lookups, then their checks and scores, all issued before use
        int j[kFoldBatch];
        bool held[kFoldBatch];
        float sc[kFoldBatch];
#pragma unroll
        for (int u = 0; u < kFoldBatch; ++u) {
            const int l = l0 + u;
            j[u] = l < a.layers ? __ldg(a.inv + ((int64_t)b * a.layers + l) * a.pos_cap + p) : -1;
        }
#pragma unroll
        for (int u = 0; u < kFoldBatch; ++u) {
            const int64_t row = (int64_t)b * a.layers + l0 + u;
            held[u] = j[u] >= 0 && j[u] < L && __ldg(a.pos + row * a.cap + j[u]) == p;
        }
        int kk = k;
#pragma unroll
        for (int u = 0; u < kFoldBatch; ++u) {
            const int l = l0 + u;
            sc[u] = 0.f;
            if (l < a.layers && a.scoring && ((a.elig_bits[l >> 5] >> (l & 31)) & 1u)) {
                if (held[u]) sc[u] = __ldg(a.sbuf + ((int64_t)b * a.n_elig + kk) * a.lstride + j[u]);
                ++kk;
            }
        }
#pragma unroll
        for (int u = 0; u < kFoldBatch; ++u) {
            const int l = l0 + u;
            if (l >= a.layers) break;
            if (a.scoring && ((a.elig_bits[l >> 5] >> (l & 31)) & 1u)) {
                m = a.alpha * m + (1.f - a.alpha) * sc[u];
                ++k;
            }
            if (held[u]) a.util[((int64_t)b * a.layers + l) * a.cap + j[u]] = m;
        }
    }
    *mp = m;
}

}  // namespace

cudaError_t launch_layer_begin(const LayerArgs &a, int32_t max_len, cudaStream_t st) {
    if (max_len > 0) {
        cudaError_t e = launch_k(layer_mark_kernel, dim3((max_len + kMarkThreads - 1) / kMarkThreads, a.layers, a.batch),
                                 dim3(kMarkThreads), 0, st, a);
        note_launch();
        if (e != cudaSuccess) return e;
    }
    cudaError_t e = launch_k(layer_begin_kernel, dim3(a.batch), dim3(kBeginThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_layer_fold(const LayerArgs &a, int32_t max_len, int32_t max_pos, cudaStream_t st) {
    if (max_len <= 0 || max_pos <= 0) return cudaSuccess;
    cudaError_t e = launch_k(layer_inverse_kernel, dim3((max_len + kInvThreads - 1) / kInvThreads, a.layers, a.batch),
                             dim3(kInvThreads), 0, st, a);
    note_launch();
    if (e != cudaSuccess) return e;
    e = launch_k(layer_fold_kernel, dim3((max_pos + kFoldThreads - 1) / kFoldThreads, a.batch), dim3(kFoldThreads), 0,
                 st, a);
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
