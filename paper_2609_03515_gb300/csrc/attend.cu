// Split-K grouped-query decode attention that also emits per-token logits.
//
// One CTA handles (split s, kv head g, sequence b, layer l): the G query heads
// of KV head g against cache slots [s*split, min((s+1)*split, len[b])).
// K/V rows stream through shared memory in 64-token tiles (cp.async, 16-byte
// chunks, XOR-swizzled by row so both the token-major QK reads and the
// dim-major PV reads are bank-conflict free).  QK: each warp owns a quarter of
// the head dimension and two tokens per lane; partial dot products meet in
// shared memory.  Softmax is online per head in the log2 domain (the query is
// pre-scaled by log2(e)/sqrt(d)); each tile's logits are written out for the
// Eq. 1 score pass.  PV: each thread owns one 16-byte column chunk of V for all
// G heads over a strided subset of the tile's tokens.  The split's running
// (max, sum) and unnormalised output go to the workspace; combine_kernel merges
// splits, writes the output and the per-head log-sum-exp.
#include "ikv_internal.cuh"

namespace ikv {
namespace {

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

template <typename T>
struct Chunk;
template <>
struct Chunk<__nv_bfloat16> {
    static constexpr int kElems = 8;
    __device__ __forceinline__ static void load(const uint4 &c, float *x) {
        const uint32_t w[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            x[2 * i] = __uint_as_float(w[i] << 16);
            x[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
        }
    }
    __device__ __forceinline__ static void store(void *p, int64_t idx, float v) {
        reinterpret_cast<__nv_bfloat16 *>(p)[idx] = __float2bfloat16_rn(v);
    }
    __device__ __forceinline__ static float read(const void *p, int64_t idx) {
        return __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(p)[idx]);
    }
};
template <>
struct Chunk<float> {
    static constexpr int kElems = 4;
    __device__ __forceinline__ static void load(const uint4 &c, float *x) {
        x[0] = __uint_as_float(c.x);
        x[1] = __uint_as_float(c.y);
        x[2] = __uint_as_float(c.z);
        x[3] = __uint_as_float(c.w);
    }
    __device__ __forceinline__ static void store(void *p, int64_t idx, float v) {
        reinterpret_cast<float *>(p)[idx] = v;
    }
    __device__ __forceinline__ static float read(const void *p, int64_t idx) {
        return reinterpret_cast<const float *>(p)[idx];
    }
};

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <typename T, int D, int G>
struct AttendCfg {
    static constexpr int TT = kTileTokens;
    static constexpr int kRowBytes = D * (int)sizeof(T);
    static constexpr int CPR = kRowBytes / 16;             // 16-byte chunks per row
    static constexpr int EPC = Chunk<T>::kElems;          // elements per chunk
    static constexpr int QCH = CPR / 4;                   // chunks per warp in QK
    static constexpr int NTG = kAttendThreads / CPR;      // token groups in PV
    static constexpr int kTileBytes = TT * kRowBytes;
    static constexpr int kStageBytes = 2 * kTileBytes;    // K + V
    static constexpr int NSTAGE = kStageBytes <= 32768 ? 3 : 2;
    static constexpr int GP = (G + 3) / 4 * 4;
    static constexpr int kStageArea = NSTAGE * kStageBytes;
    static constexpr int kObufBytes = NTG * G * D * 4;
    static_assert(kObufBytes <= kStageArea, "output reduction must fit in the stage area");
    static_assert(CPR >= 8 && CPR % 4 == 0, "row must be >= 8 chunks");
    // float regions after the stage area
    static constexpr int kQ = 0;                          // G*D
    static constexpr int kRed = kQ + G * D;               // 4*G*TT
    static constexpr int kZ = kRed + 4 * G * TT;          // G*TT
    static constexpr int kP = kZ + G * TT;                // TT*GP
    static constexpr int kM = kP + TT * GP;               // G
    static constexpr int kL = kM + GP;                    // G
    static constexpr int kC = kL + GP;                    // G
    static constexpr int kFloats = kC + GP;
    static constexpr int kSmemBytes = kStageArea + kFloats * 4;
};

template <typename T, int D, int G, bool LOGITS>
__global__ void __launch_bounds__(kAttendThreads, 2) attend_split_kernel(const AttendArgs a) {
    using C = AttendCfg<T, D, G>;
    pdl_wait();
    extern __shared__ __align__(128) unsigned char smem[];
    float *fs = reinterpret_cast<float *>(smem + C::kStageArea);
    float *q_s = fs + C::kQ;
    float *red = fs + C::kRed;
    float *zt = fs + C::kZ;
    float *p_s = fs + C::kP;
    float *m_run = fs + C::kM;
    float *l_run = fs + C::kL;
    float *corr_s = fs + C::kC;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int s = blockIdx.x, g = blockIdx.y;
    const int b = blockIdx.z % a.batch, li = blockIdx.z / a.batch;
    const int l = a.layer0 + li;
    const int L = a.len[b];
    const int S0 = a.pv.start_of(b);
    const int32_t *prow = a.pos ? a.pos + ((int64_t)b * a.rows_per_seq + (a.rows_per_seq == 1 ? 0 : g)) * a.cap : nullptr;
    const int t0 = s * a.split_tokens;
    if (t0 >= L) return;
    const int t1 = min(t0 + a.split_tokens, L);
    const int H = a.q_heads;
    const int n_tiles = (t1 - t0 + C::TT - 1) / C::TT;

    const unsigned char *kbase = reinterpret_cast<const unsigned char *>(a.k);
    const unsigned char *vbase = reinterpret_cast<const unsigned char *>(a.v);

    auto issue_tile = [&](int tile) {
        unsigned char *st = smem + (tile % C::NSTAGE) * C::kStageBytes;
        const int base = t0 + tile * C::TT;
#pragma unroll
        for (int it = 0; it < C::TT * C::CPR / kAttendThreads; ++it) {
            const int idx = it * kAttendThreads + tid;
            const int j = idx / C::CPR, c = idx % C::CPR;
            const int tok = base + j;
            if (tok < t1) {
                const int64_t row = a.pv.row_phys(b, l, g, S0 + tok);
                const int off = j * C::kRowBytes + ((c ^ (j & 7)) << 4);
                cp_async16(st + off, kbase + row * C::kRowBytes + c * 16);
                cp_async16(st + C::kTileBytes + off, vbase + row * C::kRowBytes + c * 16);
            }
        }
    };

    // prologue: start the first tiles before touching anything else
#pragma unroll
    for (int i = 0; i < C::NSTAGE - 1; ++i) {
        if (i < n_tiles) issue_tile(i);
        cp_async_commit();
    }

    // query of the G heads, pre-scaled into the log2 domain
    const int64_t qoff = (((int64_t)li * a.batch + b) * H + (int64_t)g * G) * D;
    for (int i = tid; i < G * D; i += kAttendThreads) q_s[i] = Chunk<T>::read(a.q, qoff + i) * a.scale_log2;
    if (tid < G) {
        m_run[tid] = -INFINITY;
        l_run[tid] = 0.f;
    }

    float o[G][C::EPC];
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < C::EPC; ++e) o[h][e] = 0.f;

    const int pc = tid % C::CPR;   // PV column chunk
    const int tg = tid / C::CPR;   // PV token group

    for (int tile = 0; tile < n_tiles; ++tile) {
        __syncthreads();  // previous tile's PV done with its stage and with p_s
        if (tile + C::NSTAGE - 1 < n_tiles) issue_tile(tile + C::NSTAGE - 1);
        cp_async_commit();
        cp_async_wait<C::NSTAGE - 1>();
        __syncthreads();

        const unsigned char *Ks = smem + (tile % C::NSTAGE) * C::kStageBytes;
        const unsigned char *Vs = Ks + C::kTileBytes;
        const int tbase = t0 + tile * C::TT;
        const int nv = min(C::TT, t1 - tbase);

        // ---- QK: warp owns chunks [warp*QCH, (warp+1)*QCH), lane owns tokens lane, lane+32
        {
            float acc0[G], acc1[G];
#pragma unroll
            for (int h = 0; h < G; ++h) acc0[h] = acc1[h] = 0.f;
            const int j0 = lane, j1 = lane + 32;
#pragma unroll
            for (int qc = 0; qc < C::QCH; ++qc) {
                const int c = warp * C::QCH + qc;
                float x0[C::EPC], x1[C::EPC];
                Chunk<T>::load(*reinterpret_cast<const uint4 *>(Ks + j0 * C::kRowBytes + ((c ^ (j0 & 7)) << 4)), x0);
                Chunk<T>::load(*reinterpret_cast<const uint4 *>(Ks + j1 * C::kRowBytes + ((c ^ (j1 & 7)) << 4)), x1);
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float4 *qp = reinterpret_cast<const float4 *>(q_s + h * D + c * C::EPC);
#pragma unroll
                    for (int e4 = 0; e4 < C::EPC / 4; ++e4) {
                        const float4 qv = qp[e4];
                        acc0[h] = fmaf(qv.x, x0[4 * e4 + 0], acc0[h]);
                        acc0[h] = fmaf(qv.y, x0[4 * e4 + 1], acc0[h]);
                        acc0[h] = fmaf(qv.z, x0[4 * e4 + 2], acc0[h]);
                        acc0[h] = fmaf(qv.w, x0[4 * e4 + 3], acc0[h]);
                        acc1[h] = fmaf(qv.x, x1[4 * e4 + 0], acc1[h]);
                        acc1[h] = fmaf(qv.y, x1[4 * e4 + 1], acc1[h]);
                        acc1[h] = fmaf(qv.z, x1[4 * e4 + 2], acc1[h]);
                        acc1[h] = fmaf(qv.w, x1[4 * e4 + 3], acc1[h]);
                    }
                }
            }
#pragma unroll
            for (int h = 0; h < G; ++h) {
                red[(warp * G + h) * C::TT + j0] = acc0[h];
                red[(warp * G + h) * C::TT + j1] = acc1[h];
            }
        }
        __syncthreads();

        // ---- logits of this tile (log2 domain), masked tail and dead slots (-inf)
        for (int idx = tid; idx < G * C::TT; idx += kAttendThreads) {
            const int h = idx / C::TT, j = idx % C::TT;
            float z = red[(0 * G + h) * C::TT + j] + red[(1 * G + h) * C::TT + j] + red[(2 * G + h) * C::TT + j] +
                      red[(3 * G + h) * C::TT + j];
            if (j < nv) {
                if (prow && prow[tbase + j] < 0) z = -INFINITY;
                if (LOGITS)
                    a.logits[((((int64_t)b * a.sc_layers + a.sc_layer0 + li) * H) + g * G + h) * (int64_t)a.lstride +
                             tbase + j] = z;
            } else {
                z = -INFINITY;
            }
            zt[h * C::TT + j] = z;
        }
        __syncthreads();

        // ---- online softmax per head
        for (int h = warp; h < G; h += kAttendThreads / 32) {
            const float za = zt[h * C::TT + lane], zb = zt[h * C::TT + lane + 32];
            const float mx = warp_max(fmaxf(za, zb));
            const float m_old = m_run[h];
            const float m_new = fmaxf(m_old, mx);
            const float m_ref = m_new == -INFINITY ? 0.f : m_new;  // every slot so far dead: nothing to scale
            const float corr = exp2f(m_old - m_ref);
            const float pa = exp2f(za - m_ref), pb = exp2f(zb - m_ref);
            const float sum = warp_sum(pa + pb);
            p_s[lane * C::GP + h] = pa;
            p_s[(lane + 32) * C::GP + h] = pb;
            __syncwarp();
            if (lane == 0) {
                l_run[h] = l_run[h] * corr + sum;
                m_run[h] = m_new;
                corr_s[h] = corr;
            }
        }
        __syncthreads();

        // ---- PV
        {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float cr = corr_s[h];
#pragma unroll
                for (int e = 0; e < C::EPC; ++e) o[h][e] *= cr;
            }
            for (int j = tg; j < nv; j += C::NTG) {
                float xv[C::EPC];
                Chunk<T>::load(*reinterpret_cast<const uint4 *>(Vs + j * C::kRowBytes + ((pc ^ (j & 7)) << 4)), xv);
                float p[C::GP];
#pragma unroll
                for (int h4 = 0; h4 < C::GP / 4; ++h4) {
                    const float4 pv = reinterpret_cast<const float4 *>(p_s + j * C::GP)[h4];
                    p[4 * h4] = pv.x;
                    p[4 * h4 + 1] = pv.y;
                    p[4 * h4 + 2] = pv.z;
                    p[4 * h4 + 3] = pv.w;
                }
#pragma unroll
                for (int h = 0; h < G; ++h)
#pragma unroll
                    for (int e = 0; e < C::EPC; ++e) o[h][e] = fmaf(p[h], xv[e], o[h][e]);
            }
        }
    }

    // ---- reduce the PV token groups, write the split partial
    cp_async_wait<0>();
    __syncthreads();
    float *obuf = reinterpret_cast<float *>(smem);
#pragma unroll
    for (int h = 0; h < G; ++h)
#pragma unroll
        for (int e = 0; e < C::EPC; ++e) obuf[(tg * G + h) * D + pc * C::EPC + e] = o[h][e];
    __syncthreads();
    const int64_t pbase = (((int64_t)b * a.n_layers + li) * H + (int64_t)g * G) * a.n_splits;
    for (int idx = tid; idx < G * D; idx += kAttendThreads) {
        const int h = idx / D, e = idx % D;
        float acc = 0.f;
#pragma unroll
        for (int t = 0; t < C::NTG; ++t) acc += obuf[(t * G + h) * D + e];
        a.part_o[((pbase + (int64_t)h * a.n_splits) + s) * D + e] = acc;
    }
    if (tid < G) {
        a.part_ml[((pbase + (int64_t)tid * a.n_splits) + s) * 2 + 0] = m_run[tid];
        a.part_ml[((pbase + (int64_t)tid * a.n_splits) + s) * 2 + 1] = l_run[tid];
    }
}

template <typename T>
__global__ void __launch_bounds__(128) combine_kernel(const CombineArgs a) {
    pdl_wait();
    const int h = blockIdx.x;
    const int b = blockIdx.y % a.batch, li = blockIdx.y / a.batch;
    const int D = a.head_dim;
    const int L = a.len[b];
    const int ns = min((L + a.split_tokens - 1) / a.split_tokens, a.n_splits);
    const int64_t pbase = (((int64_t)b * a.n_layers + li) * a.q_heads + h) * a.n_splits;
    const float *ml = a.part_ml + pbase * 2;
    float M = -INFINITY;
    for (int s = 0; s < ns; ++s) M = fmaxf(M, ml[2 * s]);
    const float Mref = M == -INFINITY ? 0.f : M;  // splits whose slots are all dead carry -inf
    float wsum = 0.f;
    for (int s = 0; s < ns; ++s) wsum += ml[2 * s + 1] * exp2f(ml[2 * s] - Mref);
    const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
    const int64_t obase = (((int64_t)li * a.batch + b) * a.q_heads + h) * D;
    for (int e = threadIdx.x; e < D; e += blockDim.x) {
        float acc = 0.f;
        for (int s = 0; s < ns; ++s) acc += a.part_o[(pbase + s) * D + e] * exp2f(ml[2 * s] - Mref);
        Chunk<T>::store(a.out, obase + e, acc * inv);
    }
    if (a.lse2 && threadIdx.x == 0)
        a.lse2[((int64_t)b * a.sc_layers + a.sc_layer0 + li) * a.q_heads + h] = wsum > 0.f ? M + log2f(wsum) : -INFINITY;
}

template <typename T, int D, int G>
cudaError_t launch_attend_t(const AttendArgs &a, cudaStream_t st) {
    using C = AttendCfg<T, D, G>;
    dim3 grid(a.n_splits, a.pv.kv_heads, a.batch * a.n_layers);
    if (a.logits) {
        auto k = attend_split_kernel<T, D, G, true>;
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
        if (e != cudaSuccess) return e;
        { cudaError_t le = launch_k(k, grid, dim3(kAttendThreads), C::kSmemBytes, st, a); if (le != cudaSuccess) return le; }
    } else {
        auto k = attend_split_kernel<T, D, G, false>;
        cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmemBytes);
        if (e != cudaSuccess) return e;
        { cudaError_t le = launch_k(k, grid, dim3(kAttendThreads), C::kSmemBytes, st, a); if (le != cudaSuccess) return le; }
    }
    note_launch();
    return cudaGetLastError();
}

template <typename T, int D>
cudaError_t launch_attend_d(const AttendArgs &a, int group, cudaStream_t st) {
    switch (group) {
        case 1: return launch_attend_t<T, D, 1>(a, st);
        case 2: return launch_attend_t<T, D, 2>(a, st);
        case 4: return launch_attend_t<T, D, 4>(a, st);
        case 7: return launch_attend_t<T, D, 7>(a, st);
        case 8: return launch_attend_t<T, D, 8>(a, st);
        default: return cudaErrorInvalidValue;
    }
}

}  // namespace

cudaError_t launch_attend(const AttendArgs &a, int dtype, int head_dim, int group, cudaStream_t st) {
    if (dtype == IKV_BF16) {
        if (head_dim == 128) return launch_attend_d<__nv_bfloat16, 128>(a, group, st);
        if (head_dim == 64) return launch_attend_d<__nv_bfloat16, 64>(a, group, st);
    } else {
        if (head_dim == 128) return launch_attend_d<float, 128>(a, group, st);
        if (head_dim == 64) return launch_attend_d<float, 64>(a, group, st);
    }
    return cudaErrorInvalidValue;
}

cudaError_t launch_combine(const CombineArgs &a, int dtype, cudaStream_t st) {
    dim3 grid(a.q_heads, a.batch * a.n_layers);
    if (dtype == IKV_BF16)
        { cudaError_t le = launch_k(combine_kernel<__nv_bfloat16>, grid, dim3(128), 0, st, a); if (le != cudaSuccess) return le; }
    else
        { cudaError_t le = launch_k(combine_kernel<float>, grid, dim3(128), 0, st, a); if (le != cudaSuccess) return le; }
    note_launch();
    return cudaGetLastError();
}

}  // namespace ikv
