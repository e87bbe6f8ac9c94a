// Rank-trace diagnostics (Appendix "Mechanistic Diagnostics"): per utility row, the
// raw top-k set (the step's single-step score, before eviction) and the EMA top-k set
// (the tokens kept), as sorted token positions, and their overlaps with each other and
// with the previous traced step's sets.
#include <climits>

#include "ikv_internal.cuh"

namespace ikv {

__device__ unsigned int g_trace_error = 0;  // bit 4: a set exceeded kTraceMax tokens

namespace {

constexpr int kTraceMax = 16384;   // tokens per set sorted in shared memory
constexpr int kTraceThreads = 1024;

__global__ void trace_gather_kernel(const TraceArgs a) {
    pdl_wait();
    const int r = blockIdx.y;
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const int n = a.n_raw[r];
    if (j < n) a.raw_pos[(int64_t)r * a.cap + j] = a.pos[(int64_t)r * a.cap + a.keep_raw[(int64_t)r * a.cap + j]];
}

// ascending bitonic sort of n2 (a power of two) ints in shared memory
__device__ void bitonic_sort(int *x, int n2) {
    for (int k = 2; k <= n2; k <<= 1)
        for (int j = k >> 1; j > 0; j >>= 1) {
            for (int i = threadIdx.x; i < n2; i += blockDim.x) {
                const int o = i ^ j;
                if (o > i) {
                    const bool up = (i & k) == 0;
                    const int u = x[i], v = x[o];
                    if ((u > v) == up) {
                        x[i] = v;
                        x[o] = u;
                    }
                }
            }
            __syncthreads();
        }
}

__device__ __forceinline__ bool contains(const int *x, int n, int v) {
    int lo = 0, hi = n;
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (x[mid] < v) lo = mid + 1;
        else hi = mid;
    }
    return lo < n && x[lo] == v;
}

__device__ __forceinline__ int pow2_at_least(int n) {
    int p = 1;
    while (p < n) p <<= 1;
    return p;
}

// One CTA per utility row.
__global__ void __launch_bounds__(kTraceThreads) trace_kernel(const TraceArgs a) {
    pdl_wait();
    extern __shared__ int tsm[];
    int *Rs = tsm, *Es = tsm + kTraceMax;
    __shared__ int nE_s, c_rr, c_ee, c_re;
    const int r = blockIdx.x, tid = threadIdx.x;
    const int b = r / a.rows_per_seq;
    const int L = a.len[b];
    if (tid == 0) nE_s = c_rr = c_ee = c_re = 0;
    __syncthreads();
    const int32_t *pr = a.pos + (int64_t)r * a.cap;
    for (int j = tid; j < L; j += kTraceThreads) {
        const int p = pr[j];
        if (p >= 0) {
            const int i = atomicAdd(&nE_s, 1);
            if (i < kTraceMax) Es[i] = p;
        }
    }
    __syncthreads();
    const int nE = nE_s;
    const int nR = a.has_raw ? a.n_raw[r] : 0;
    if (nE > kTraceMax || nR > kTraceMax) {
        if (tid == 0) {
            atomicOr(&g_trace_error, 16u);
            for (int k = 0; k < 5; ++k) a.counts[(int64_t)r * 5 + k] = -2;
        }
        return;
    }
    const int pE = pow2_at_least(nE), pR = pow2_at_least(nR);
    for (int i = tid; i < pE; i += kTraceThreads)
        if (i >= nE) Es[i] = INT_MAX;
    for (int i = tid; i < pR; i += kTraceThreads) Rs[i] = i < nR ? a.raw_pos[(int64_t)r * a.cap + i] : INT_MAX;
    __syncthreads();
    bitonic_sort(Es, pE);
    bitonic_sort(Rs, pR);
    const int *prevR = a.raw_top + (int64_t)r * a.cap, *prevE = a.ema_top + (int64_t)r * a.cap;
    const int nPR = a.n_top[2 * r], nPE = a.n_top[2 * r + 1];
    int rr = 0, ee = 0, re = 0;
    for (int i = tid; i < nR; i += kTraceThreads) {
        rr += contains(prevR, nPR, Rs[i]);
        re += contains(Es, nE, Rs[i]);
    }
    for (int i = tid; i < nE; i += kTraceThreads) ee += contains(prevE, nPE, Es[i]);
    if (rr) atomicAdd(&c_rr, rr);
    if (ee) atomicAdd(&c_ee, ee);
    if (re) atomicAdd(&c_re, re);
    __syncthreads();  // every read of the previous sets is done before they are replaced
    if (tid == 0) {
        int *c = a.counts + (int64_t)r * 5;
        c[0] = a.has_raw ? c_rr : -1;
        c[1] = c_ee;
        c[2] = a.has_raw ? c_re : -1;
        c[3] = a.has_raw ? nR : -1;
        c[4] = nE;
        if (a.has_raw) a.n_top[2 * r] = nR;
        a.n_top[2 * r + 1] = nE;
    }
    if (a.has_raw)
        for (int i = tid; i < nR; i += kTraceThreads) a.raw_top[(int64_t)r * a.cap + i] = Rs[i];
    for (int i = tid; i < nE; i += kTraceThreads) a.ema_top[(int64_t)r * a.cap + i] = Es[i];
}

}  // namespace

cudaError_t launch_trace_gather(const TraceArgs &a, int32_t max_len, cudaStream_t st) {
    if (max_len <= 0 || a.rows <= 0) return cudaSuccess;
    cudaError_t e = launch_k(trace_gather_kernel, dim3((max_len + 255) / 256, a.rows), dim3(256), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_trace(const TraceArgs &a, cudaStream_t st) {
    if (a.rows <= 0) return cudaSuccess;
    constexpr size_t smem = 2 * kTraceMax * sizeof(int);
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(trace_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    cudaError_t e = launch_k(trace_kernel, dim3(a.rows), dim3(kTraceThreads), smem, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t read_clear_trace_error(unsigned int *v) {
    unsigned int z = 0;
    cudaError_t e = cudaMemcpyFromSymbol(v, g_trace_error, sizeof(*v));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_trace_error, &z, sizeof(z));
    return e;
}

}  // namespace ikv
