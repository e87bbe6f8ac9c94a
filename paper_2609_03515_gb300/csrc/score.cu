// Eq. 1 score and the layer-sequential aggregation of Eq. 2-4 (Appendix "Layer
// scoring"), fused with the softmax normalisation; the VNorm and entropy-weighted
// scorers of the Appendix "Per-step scoring"; value-row norms for VNorm.
//
// score_kernel: one 256-thread CTA per (32 V tokens, utility row, layer group): each
// group holds up to 8 consecutive eligible layers, one warp per layer, V consecutive
// tokens per lane.  Warp l computes s_l(i) = mean over the row's heads of p_h(i) =
// exp2(z_h(i) - lse2_h) from the attention kernel's log2-domain logits and log-sum-exp
// (VNorm: each head's p_h(i) times its KV head's value-norm weight).  Each update of
// Eq. 2-4 is an affine map of the utility, m -> a m + c, so a group folds its layers, in
// ascending order, into one such map per token; the last CTA of the row to finish
// applies the groups' maps to every utility in layer order (with one group each CTA runs
// the plain layer-by-layer fold itself) and, in a step, selects the row.  Splitting the
// layers over CTAs spreads a short cache over every SM, and one arrival per CTA keeps
// the chain of dependent steps after the loads short.  The entropy scorer needs every
// token of a layer before its weight is known,
// so its first pass only stores s_l and per-block partial entropies, and
// entropy_fold_kernel applies the weights and folds.
#include "ikv_internal.cuh"
#include "select_row.cuh"

namespace ikv {
namespace {

constexpr int kScoreWarps = kScoreLayersPerGroup;  // one warp per eligible layer of a layer group
constexpr int kScoreThreads = kScoreWarps * 32;    // also the fused selection's CTA size

template <int V> struct VecF;
template <> struct VecF<1> { using T = float; };
template <> struct VecF<2> { using T = float2; };
template <> struct VecF<4> { using T = float4; };
__device__ __forceinline__ float vget(float x, int) { return x; }
__device__ __forceinline__ float vget(float2 x, int v) { return v == 0 ? x.x : x.y; }
__device__ __forceinline__ float vget(float4 x, int v) { return v == 0 ? x.x : v == 1 ? x.y : v == 2 ? x.z : x.w; }

__device__ __forceinline__ float aggregate(float m, float s, int agg, float alpha) {
    if (agg == IKV_AGG_EMA) return alpha * m + (1.f - alpha) * s;  // Eq. 4
    if (agg == IKV_AGG_CUMULATIVE) return m + s;                    // Eq. 3
    return s;                                                       // Eq. 2
}
// the factor a of the affine map m -> a m + c that n consecutive updates compose to
__device__ __forceinline__ float agg_factor(int n, int agg, float alpha) {
    if (agg == IKV_AGG_CUMULATIVE) return 1.f;
    if (agg != IKV_AGG_EMA) return n > 0 ? 0.f : 1.f;
    float f = 1.f;
    for (int k = 0; k < n; ++k) f *= alpha;
    return f;
}

// thread-block cluster: barrier over every thread of the cluster (release / acquire), and a
// load from the shared memory of the cluster's CTA `rank` at the address of `p` in this one
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ float ld_cluster_f32(const float *p, int rank) {
    const uint32_t a = static_cast<uint32_t>(__cvta_generic_to_shared(p));
    uint32_t ra;
    float v;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(ra) : "r"(a), "r"(rank));
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(ra) : "memory");
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// The pass is latency bound: every head of a batch of 32 / V is loaded before any
// is used, the per-head log-sum-exp travels by shuffle, and the utility is fetched
// before the loads.  V > 1 reads each head row in 256- or 512-byte runs, which DRAM
// serves far better than scattered 128-byte pieces.
template <int V, int SCORER>
__global__ void __launch_bounds__(kScoreThreads, 4) score_kernel(const ScoreArgs a) {
    using VT = typename VecF<V>::T;
    pdl_wait();
    constexpr int kTok = 32 * V;   // tokens per CTA
    constexpr int kHB = 32 / V;    // heads per load batch (32 registers of loads)
    __shared__ __align__(16) float sl[kScoreWarps][kTok];
    extern __shared__ float wsm[];  // VNorm: per warp, [row's kv heads][kTok] value-norm weights
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.y;
    const int lg = blockIdx.z, n_lg = gridDim.z;  // this CTA's layer group, and how many there are
    const int b = r / a.rows_per_seq;
    // The row's length decides which tokens count, not which addresses are read (rows of
    // the logits and the utility are padded past every block), so the loads below do not
    // wait for it; a block past the length leaves once they are issued.
    const int L = a.len[b];
    const int i0 = blockIdx.x * kTok;
    const int il = i0 + lane * V;  // first token of this lane
    int h0 = 0, nh = a.q_heads;
    if (a.rows_per_seq > 1) {
        nh = a.q_heads / a.kv_heads;
        h0 = (r % a.rows_per_seq) * nh;
    }
    const int H = a.q_heads, G = a.q_heads / a.kv_heads;
    const float inv = 1.f / (float)nh;
    const int fi = i0 + (int)threadIdx.x;  // token folded by this thread (threads < kTok)
    const bool folds = threadIdx.x < kTok && fi < L;
    const int64_t at = (int64_t)r * a.cap + fi;
    const int kw0 = lg * kScoreWarps;                        // the group's first eligible layer (pass index)
    const int n_here = min(kScoreWarps, a.n_elig - kw0);     // layers of this group
    float m = 0.f;
    if (SCORER != IKV_SCORE_ENTROPY && threadIdx.x < kTok && fi < a.cap && a.ema) m = a.ema[at];
    if (warp < n_here) {
        const int li = a.elig[kw0 + warp];
        // row padding keeps i0 + kTok <= lstride, so the vector loads stay inside the row
        const float *zp = a.logits + (((int64_t)b * a.n_layers + li) * H + h0) * (int64_t)a.lstride + il;
        const float *ll = a.lse2 + ((int64_t)b * a.n_layers + li) * H + h0;
        const int g0 = h0 / G, ng = (nh + G - 1) / G;  // the row's kv heads
        float *wv = wsm + (size_t)warp * ng * kTok;
        if (SCORER == IKV_SCORE_VNORM) {
            // every weight this warp needs, in one batch of loads: norm over the unit's mean norm
            for (int gg = 0; gg < ng; ++gg) {
                const int g = g0 + gg;
                const float mean = a.vmean[((int64_t)b * a.n_layers + li) * a.kv_heads + g];
                const float *vn = a.vnorm + (((int64_t)(a.layer0 + li) * a.batch + b) * a.kv_heads + g) * a.cap;
#pragma unroll
                for (int v = 0; v < V; ++v)
                    wv[gg * kTok + lane * V + v] = mean > 0.f ? (il + v < L ? __ldg(vn + il + v) : 0.f) / mean : 1.f;
            }
            __syncwarp();
        }
        float acc[V];
#pragma unroll
        for (int v = 0; v < V; ++v) acc[v] = 0.f;
        // rows: the heads' log2-domain logits (normalised here by their log-sum-exp), or with
        // gsum one row per KV head of the utility row holding its query group's normalised
        // probabilities already summed
        const int nrows = a.gsum ? ng : nh;
        if (a.gsum) zp = a.logits + (((int64_t)b * a.n_layers + li) * a.kv_heads + g0) * (int64_t)a.lstride + il;
        for (int hb = 0; hb < nrows; hb += kHB) {
            const int nb = min(kHB, nrows - hb);
            const float lse_lane = !a.gsum && lane < nb ? ll[hb + lane] : 0.f;
            VT z[kHB];
#pragma unroll
            for (int j = 0; j < kHB; ++j) {
                if (j < nb) z[j] = __ldg(reinterpret_cast<const VT *>(zp));
                zp += a.lstride;
            }
            // each row's probabilities times the VNorm weight (1 for the other scorers)
            auto weight = [&](int j, float *w) {
#pragma unroll
                for (int v = 0; v < V; ++v) w[v] = 1.f;
                if (SCORER == IKV_SCORE_VNORM) {
                    const int gr = a.gsum ? hb + j : (h0 + hb + j) / G - g0;  // the row's kv head
                    const float *wg = wv + gr * kTok + lane * V;
#pragma unroll
                    for (int v = 0; v < V; ++v) w[v] = wg[v];
                }
            };
            if (a.gsum) {
#pragma unroll
                for (int j = 0; j < kHB; ++j)
                    if (il < L && j < nb) {
                        float w[V];
                        weight(j, w);
#pragma unroll
                        for (int v = 0; v < V; ++v) acc[v] += vget(z[j], v) * w[v];
                    }
            } else {
#pragma unroll
                for (int j = 0; j < kHB; ++j) {
                    const float lj = __shfl_sync(0xffffffffu, lse_lane, j);
                    if (il < L && j < nb) {
                        float w[V];
                        weight(j, w);
#pragma unroll
                        for (int v = 0; v < V; ++v) acc[v] += exp2f(vget(z[j], v) - lj) * w[v];
                    }
                }
            }
        }
#pragma unroll
        for (int v = 0; v < V; ++v) sl[warp][lane * V + v] = acc[v] * inv;
        if (SCORER != IKV_SCORE_ENTROPY && a.store_only) {  // each layer's pooled score, unfolded
            const int k = a.k0 + kw0 + warp;
#pragma unroll
            for (int v = 0; v < V; ++v)
                if (il + v < L) a.sbuf[((int64_t)r * a.n_elig_total + k) * a.lstride + il + v] = acc[v] * inv;
        }
        if (SCORER == IKV_SCORE_ENTROPY) {
            // the layer's pooled scores, and this block's share of -sum s ln s over them
            const int k = a.k0 + kw0 + warp;
            float e = 0.f;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int i = il + v;
                const float s = acc[v] * inv;
                if (i < L) {
                    a.sbuf[((int64_t)r * a.n_elig_total + k) * a.lstride + i] = s;
                    if (s > 0.f) e -= s * logf(s);
                }
            }
            e = warp_sum(e);
            if (lane == 0) a.epart[((int64_t)r * (a.n_elig_total + 1) + k) * a.nblk + blockIdx.x] = e;
        }
    }
    if (i0 >= L) return;  // every CTA of a cluster (one token block) leaves together
    if (SCORER == IKV_SCORE_ENTROPY) {
        if (warp == 0 && lg == 0) {  // live slots of this block (the entropy normalisation is ln of their count)
            float c = 0.f;
#pragma unroll
            for (int v = 0; v < V; ++v) {
                const int i = il + v;
                if (i < L && (!a.pos || a.pos[(int64_t)r * a.cap + i] >= 0)) c += 1.f;
            }
            c = warp_sum(c);
            if (lane == 0) a.epart[((int64_t)r * (a.n_elig_total + 1) + a.n_elig_total) * a.nblk + blockIdx.x] = c;
        }
        return;
    }
    if (a.store_only) return;
    __syncthreads();
    // Fold this CTA's layers for its tokens.  One group: the plain layer-by-layer fold onto
    // the utility.  Several: the group's layers as one affine map m -> f m + c (c: the fold
    // from zero); the token block's groups form one cluster, and its first CTA applies the
    // groups' maps in layer order, reading the others' c from their shared memory.
    __shared__ float cpart[kTok];
    float sc = 0.f;  // the last eligible layer's score (with one layer: the step's score)
    float c = n_lg == 1 ? m : 0.f;
    if (folds) {
        for (int k = 0; k < n_here; ++k) {
            sc = sl[k][threadIdx.x];
            c = aggregate(c, sc, a.agg, a.alpha);
        }
        if (a.score && lg == n_lg - 1) a.score[at] = sc;
    }
    if (n_lg > 1) {
        if (threadIdx.x < kTok) cpart[threadIdx.x] = c;
        cluster_sync();  // every group's c is in its shared memory
        if (lg == 0 && folds) {
            // every group's c is loaded before any is used, so the remote loads overlap
            constexpr int kMaxGroups = (kMaxLayersPerScorePass + kScoreWarps - 1) / kScoreWarps;
            float cq[kMaxGroups];
#pragma unroll
            for (int q = 1; q < kMaxGroups; ++q) cq[q] = q < n_lg ? ld_cluster_f32(&cpart[threadIdx.x], q) : 0.f;
            cq[0] = c;
#pragma unroll
            for (int q = 0; q < kMaxGroups; ++q)
                if (q < n_lg) m = agg_factor(min(kScoreWarps, a.n_elig - q * kScoreWarps), a.agg, a.alpha) * m + cq[q];
        }
        cluster_sync();  // the first CTA has read them: the others may exit
        if (lg != 0) return;
    } else {
        m = c;
    }
    if (folds && a.ema) a.ema[at] = m;
    if (!a.fuse_select) return;
    // The selection's first pass for this block: its live slots and their lowest (key,
    // highest slot), left for the row's last block to arrive
    __shared__ unsigned long long red_best[kScoreWarps];
    __shared__ uint32_t red_cnt[kScoreWarps];
    auto block_reduce = [&](uint32_t cn, unsigned long long best) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            cn += __shfl_xor_sync(0xffffffffu, cn, o);
            const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
            best = y < best ? y : best;
        }
        if (lane == 0) {
            red_best[warp] = best;
            red_cnt[warp] = cn;
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            for (int w = 1; w < kScoreWarps; ++w) {
                best = red_best[w] < best ? red_best[w] : best;
                cn += red_cnt[w];
            }
            red_best[0] = best;
            red_cnt[0] = cn;
        }
        __syncthreads();
    };
    const int blocks = (L + kTok - 1) / kTok;
    {
        uint32_t cn = 0u;
        unsigned long long best = ~0ull;
        if (folds && (!a.sel_pos || a.sel_pos[at] >= 0)) {
            cn = 1u;
            best = ((unsigned long long)ord_key(m) << 32) | (uint32_t)(~(uint32_t)fi);
        }
        block_reduce(cn, best);
        if (threadIdx.x == 0) {
            a.sel_best[(int64_t)r * a.nblk + blockIdx.x] = red_best[0];
            a.sel_cnt[(int64_t)r * a.nblk + blockIdx.x] = red_cnt[0];
        }
    }
    // every token block of the row arrives once its stores are out; the last one selects the
    // row (arrival counter only: no CTA waits for another)
    __shared__ int last;
    __syncthreads();
    if (threadIdx.x == 0) {
        last = arrive_acq_rel(a.row_done + r) == blocks - 1;
        if (last) a.row_done[r] = 0;
    }
    __syncthreads();
    if (!last) return;
    // the blocks' partials give the live count and the victim candidate
    uint32_t cn = 0u;
    unsigned long long best = ~0ull;
    for (int jb = threadIdx.x; jb < blocks; jb += kScoreThreads) {
        const unsigned long long y = __ldcg(a.sel_best + (int64_t)r * a.nblk + jb);
        best = y < best ? y : best;
        cn += __ldcg(a.sel_cnt + (int64_t)r * a.nblk + jb);
    }
    block_reduce(cn, best);
    const unsigned long long s_best = red_best[0];
    const int n_live = (int)red_cnt[0];
    const int B = max(a.budget[b], 0);
    const int S = a.df.start ? a.df.start[b] : 0;
    if (a.sel_pos && a.df.max_holes > 0 && B > 0 && n_live == B + 1 && L - B <= a.df.max_holes && S + L < a.df.cap) {
        // one slot too many and the sequence may defer: mark the victim dead, as the
        // selection itself would
        if (threadIdx.x == 0) {
            a.sel_pos[(int64_t)r * a.cap + (int)(~(uint32_t)(s_best & 0xFFFFFFFFull))] = -1;
            a.keep_len[r] = -1 - B;
        }
    } else {
        select_row<kScoreThreads>(r, a.cap, a.ema, a.len, a.rows_per_seq, a.budget, a.sel_pos, a.keep, a.keep_len,
                                  a.df);
    }
}

// Entropy weighting, second pass: the normalised entropy w_k = H(s_k) / ln n of every
// eligible layer's pooled score distribution (n live slots; 1 when n <= 1), then the
// layer-sequential fold of w_k s_k(i) for this CTA's tokens.
constexpr int kFoldThreads = 256;
__global__ void __launch_bounds__(kFoldThreads) entropy_fold_kernel(const ScoreArgs a) {
    pdl_wait();
    __shared__ float wk[kMaxLayers];
    __shared__ float n_live;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int r = blockIdx.y;
    const int L = a.len[r / a.rows_per_seq];
    const int i = blockIdx.x * kFoldThreads + threadIdx.x;
    if ((int)(blockIdx.x * kFoldThreads) >= L) return;
    const int NE = a.n_elig_total;
    const float *ep = a.epart + (int64_t)r * (NE + 1) * a.nblk;
    const int nb = (L + a.blk_tok - 1) / a.blk_tok;  // the blocks the first pass wrote for this row
    if (warp == 0) {
        float c = 0.f;
        for (int j = lane; j < nb; j += 32) c += ep[(int64_t)NE * a.nblk + j];
        c = warp_sum(c);
        if (lane == 0) n_live = c;
    }
    __syncthreads();
    const float n = n_live;
    for (int k = warp; k < NE; k += kFoldThreads / 32) {
        float e = 0.f;
        for (int j = lane; j < nb; j += 32) e += ep[(int64_t)k * a.nblk + j];
        e = warp_sum(e);
        if (lane == 0) wk[k] = n > 1.5f ? e / logf(n) : 1.f;
    }
    __syncthreads();
    if (i >= L) return;
    const int64_t at = (int64_t)r * a.cap + i;
    float m = a.ema[at];
    for (int k0 = 0; k0 < NE; k0 += 16) {  // 16 layers' scores in flight, then folded in order
        float sv[16];
#pragma unroll
        for (int u = 0; u < 16; ++u) sv[u] = k0 + u < NE ? a.sbuf[((int64_t)r * NE + k0 + u) * a.lstride + i] : 0.f;
#pragma unroll
        for (int u = 0; u < 16; ++u)
            if (k0 + u < NE) m = aggregate(m, wk[k0 + u] * sv[u], a.agg, a.alpha);
    }
    a.ema[at] = m;
}

// Mean value-row norm of every (sequence, layer, kv head) over its live slots.
constexpr int kMeanThreads = 256;
__global__ void __launch_bounds__(kMeanThreads) vnorm_mean_kernel(const ScoreArgs a) {
    pdl_wait();
    __shared__ float red[2][kMeanThreads / 32];
    const int u = blockIdx.x;  // (b * n_layers + li) * kv_heads + g
    const int g = u % a.kv_heads, li = (u / a.kv_heads) % a.n_layers, b = u / a.kv_heads / a.n_layers;
    const int L = a.len[b];
    const int r = b * a.rows_per_seq + (a.rows_per_seq == 1 ? 0 : g);
    const float *vn = a.vnorm + (((int64_t)(a.layer0 + li) * a.batch + b) * a.kv_heads + g) * a.cap;
    float s = 0.f, c = 0.f;
    for (int i = threadIdx.x; i < L; i += kMeanThreads)
        if (!a.pos || a.pos[(int64_t)r * a.cap + i] >= 0) {
            s += vn[i];
            c += 1.f;
        }
    s = warp_sum(s);
    c = warp_sum(c);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (lane == 0) red[0][warp] = s, red[1][warp] = c;
    __syncthreads();
    if (threadIdx.x == 0) {
        float ts = 0.f, tc = 0.f;
        for (int w = 0; w < kMeanThreads / 32; ++w) ts += red[0][w], tc += red[1][w];
        a.vmean[u] = tc > 0.f ? ts / tc : 0.f;
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

// l2 norm of every cached value row: one warp per (layer, sequence, kv head, slot).
template <typename T>
__global__ void value_norms_kernel(const T *v, PagedView pv, const int32_t *len, int32_t batch, int32_t layers,
                                   int32_t cap, float *vnorm) {
    const int lane = threadIdx.x & 31;
    const int64_t wid = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const int64_t units = (int64_t)layers * batch * pv.kv_heads;
    const int64_t u = wid / cap;
    const int j = (int)(wid % cap);
    if (u >= units) return;
    const int g = (int)(u % pv.kv_heads), b = (int)((u / pv.kv_heads) % batch), l = (int)(u / pv.kv_heads / batch);
    if (j >= len[b]) return;
    const T *row = v + pv.row_phys(b, l, g, pv.start_of(b) + j) * pv.head_dim;
    float s = 0.f;
    for (int e = lane; e < pv.head_dim; e += 32) {
        const float x = static_cast<float>(row[e]);
        s += x * x;
    }
    s = warp_sum(s);
    if (lane == 0) vnorm[u * cap + j] = sqrtf(s);
}

}  // namespace

// VNorm weight staging: per warp, one kTok-token row per kv head of the utility row
static size_t vnorm_smem(const ScoreArgs &a, int V) {
    const int ng = a.rows_per_seq > 1 ? 1 : a.kv_heads;
    return (size_t)kScoreWarps * ng * 32 * V * sizeof(float);
}
constexpr size_t kVnormSmemMax = 160 * 1024;

int score_layer_groups(int n_elig) {
    const int n = n_elig < kMaxLayersPerScorePass ? n_elig : kMaxLayersPerScorePass;
    return n <= 0 ? 1 : (n + kScoreWarps - 1) / kScoreWarps;
}

int score_blocks(const ScoreArgs &a, int32_t max_len, int sms, int *V) {
    // widest token vector that still gives every SM two CTAs (over all layer groups)
    const int64_t rows = (int64_t)a.batch * a.rows_per_seq * score_layer_groups(a.n_elig_total);
    auto ctas = [&](int tok) { return rows * ((max_len + tok - 1) / tok); };
    int v = ctas(128) >= 2 * sms ? 4 : ctas(64) >= 2 * sms ? 2 : 1;
    if (a.scorer == IKV_SCORE_VNORM)  // the weight staging must fit in shared memory
        while (v > 1 && vnorm_smem(a, v) > kVnormSmemMax) v >>= 1;
    *V = v;
    return (max_len + 32 * v - 1) / (32 * v);
}

// Shared memory a score CTA reserves so that no more than k CTAs share an SM, when the
// whole grid fits at k per SM for some k < 4 (four fit by registers).  Left to itself the
// block scheduler puts four CTAs on some SMs and one on others, and the most loaded SM
// sets the pass's pace (config 1: 412 CTAs; with at most three per SM the graphed step
// measured 81.7 -> 80.8 us).  Each size admits exactly k CTAs of this kernel (its static
// shared memory and the 1 KB reserved per CTA included) in an SM's 228 KB.
static size_t spread_smem(int64_t ctas, int sms) {
    const int64_t k = sms > 0 ? (ctas + sms - 1) / sms : 4;
    if (k >= 4 || k < 1) return 0;
    return k == 3 ? 60 * 1024 : k == 2 ? 100 * 1024 : 150 * 1024;
}
constexpr size_t kScoreSmemAttr = 180 * 1024;  // dynamic shared-memory limit set once per instantiation
static_assert(kVnormSmemMax <= kScoreSmemAttr, "VNorm staging within the limit");

// The layer groups of a token block (grid z) run as one cluster.
template <int V, int SCORER>
static cudaError_t launch_score_v(const ScoreArgs &a, dim3 grid, size_t reserve, cudaStream_t st) {
    size_t smem = SCORER == IKV_SCORE_VNORM ? vnorm_smem(a, V) : 0;
    if (smem < reserve) smem = reserve;
    static bool limit_set = false;
    if (!limit_set) {
        cudaError_t e = cudaFuncSetAttribute(score_kernel<V, SCORER>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kScoreSmemAttr);
        if (e != cudaSuccess) return e;
        limit_set = true;
    }
    if (grid.z == 1) return launch_k(score_kernel<V, SCORER>, grid, dim3(kScoreThreads), smem, st, a);
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kScoreThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = grid.z;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, score_kernel<V, SCORER>, a);
}

template <int SCORER>
static cudaError_t launch_score_t(const ScoreArgs &a, dim3 grid, int V, size_t reserve, cudaStream_t st) {
    if (V == 4) return launch_score_v<4, SCORER>(a, grid, reserve, st);
    if (V == 2) return launch_score_v<2, SCORER>(a, grid, reserve, st);
    return launch_score_v<1, SCORER>(a, grid, reserve, st);
}

cudaError_t launch_score_ema(const ScoreArgs &a, int32_t max_len, int sms, cudaStream_t st) {
    if (max_len <= 0 || a.n_elig <= 0) return cudaSuccess;
    int V = 1;
    const int nblk = score_blocks(a, max_len, sms, &V);
    const int n_lg = score_layer_groups(a.n_elig);
    dim3 grid(nblk, (unsigned)(a.batch * a.rows_per_seq), (unsigned)n_lg);
    const size_t reserve = spread_smem((int64_t)grid.x * grid.y * grid.z, sms);
    cudaError_t e;
    if (a.scorer == IKV_SCORE_VNORM)
        e = launch_score_t<IKV_SCORE_VNORM>(a, grid, V, reserve, st);
    else if (a.scorer == IKV_SCORE_ENTROPY)
        e = launch_score_t<IKV_SCORE_ENTROPY>(a, grid, V, reserve, st);
    else
        e = launch_score_t<IKV_SCORE_ATTENTION>(a, grid, V, reserve, st);
    if (e != cudaSuccess) return e;
    note_launch();
    return cudaGetLastError();
}

cudaError_t launch_entropy_fold(const ScoreArgs &a, int32_t max_len, cudaStream_t st) {
    if (max_len <= 0 || a.n_elig_total <= 0) return cudaSuccess;
    dim3 grid((max_len + kFoldThreads - 1) / kFoldThreads, (unsigned)(a.batch * a.rows_per_seq));
    cudaError_t e = launch_k(entropy_fold_kernel, grid, dim3(kFoldThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_vnorm_mean(const ScoreArgs &a, cudaStream_t st) {
    const int units = a.batch * a.n_layers * a.kv_heads;
    if (units <= 0) return cudaSuccess;
    cudaError_t e = launch_k(vnorm_mean_kernel, dim3(units), dim3(kMeanThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_value_norms(const void *v, const PagedView &pv, const int32_t *len, int32_t batch, int32_t layers,
                               int32_t cap, int dtype, float *vnorm, cudaStream_t st) {
    const int64_t warps = (int64_t)layers * batch * pv.kv_heads * cap;
    if (warps <= 0) return cudaSuccess;
    const int64_t blocks = (warps + 7) / 8;
    if (dtype == IKV_BF16)
        value_norms_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, st>>>(
            reinterpret_cast<const __nv_bfloat16 *>(v), pv, len, batch, layers, cap, vnorm);
    else
        value_norms_kernel<float><<<(unsigned)blocks, 256, 0, st>>>(reinterpret_cast<const float *>(v), pv, len,
                                                                    batch, layers, cap, vnorm);
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
