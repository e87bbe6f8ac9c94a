// Device side of the synthetic workload generator (recipe in ikvgen.h).
// Fills a paged K/V pool with a prefilled context and produces the per-step
// appended tokens directly in HBM, so multi-GB workloads never cross PCIe.
// Every element equals the host generator's bit for bit.
#include <cuda_runtime.h>
#include <stdint.h>

#include "ikvgen.h"

namespace {

template <int DT>
__device__ __forceinline__ void put(void *out, int64_t idx, float v) {
    if (DT == IKVGEN_BF16)
        reinterpret_cast<uint16_t *>(out)[idx] = ikvgen_bf16_bits(v);
    else
        reinterpret_cast<float *>(out)[idx] = v;
}

// one thread per (row, element); rows = (b, l, g, slot) of the paged pool
template <int DT>
__global__ void fill_paged_kernel(ikvgen_spec s, const float *__restrict__ u, void *kpool, void *vpool,
                                  const int32_t *__restrict__ block_table, const int32_t *__restrict__ L0,
                                  int32_t num_pages, int32_t page_size, int32_t max_pages, int32_t max_len) {
    const int32_t d = s.head_dim;
    const int32_t b = blockIdx.z;
    const int32_t l = blockIdx.y / s.kv_heads;
    const int32_t g = blockIdx.y % s.kv_heads;
    const int64_t n_elem = (int64_t)L0[b] * d;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n_elem; i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t p = i / d;
        const int32_t e = (int32_t)(i % d);
        const int32_t page = block_table[(int64_t)b * max_pages + p / page_size];
        const int64_t row = (((int64_t)l * num_pages + page) * s.kv_heads + g) * page_size + p % page_size;
        const int heavy = ikvgen_is_heavy(&s, b, p);
        const float ue = u[((int64_t)l * s.kv_heads + g) * d + e];
        if (kpool) put<DT>(kpool, row * d + e, ikvgen_key_elem(&s, b, l, g, p, e, heavy, ue));
        if (vpool) put<DT>(vpool, row * d + e, ikvgen_value_elem(&s, b, l, g, p, e));
    }
    (void)max_len;
}

// appended tokens for steps t in [t0, t1): out [t1-t0][layers][batch][kv_heads][d]; position L0[b] + t - 1
template <int DT>
__global__ void fill_tokens_kernel(ikvgen_spec s, const float *__restrict__ u, const int32_t *__restrict__ L0,
                                   int32_t t0, int32_t t1, void *out_k, void *out_v) {
    const int32_t d = s.head_dim;
    const int64_t per_step = (int64_t)s.layers * s.batch * s.kv_heads * d;
    const int64_t n = (int64_t)(t1 - t0) * per_step;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        const int32_t ti = (int32_t)(i / per_step);
        int64_t r = i % per_step;
        const int32_t e = (int32_t)(r % d);
        r /= d;
        const int32_t g = (int32_t)(r % s.kv_heads);
        r /= s.kv_heads;
        const int32_t b = (int32_t)(r % s.batch);
        const int32_t l = (int32_t)(r / s.batch);
        const int64_t p = (int64_t)L0[b] + (t0 + ti) - 1;
        const int heavy = ikvgen_is_heavy(&s, b, p);
        const float ue = u[((int64_t)l * s.kv_heads + g) * d + e];
        if (out_k) put<DT>(out_k, i, ikvgen_key_elem(&s, b, l, g, p, e, heavy, ue));
        if (out_v) put<DT>(out_v, i, ikvgen_value_elem(&s, b, l, g, p, e));
    }
}

__global__ void normals_kernel(uint64_t seed, uint64_t stream, int64_t n, float *out) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = ikvgen_normal(seed, stream, (uint64_t)i, 0);
}

}  // namespace

extern "C" {

// Prefill positions [0, L0[b]) of every (b, layer, kv head) of a paged pool
// [layers][num_pages][kv_heads][page_size][d]. u, block_table, L0 are device pointers.
int ikvgen_fill_paged_cuda(const ikvgen_spec *spec, const float *u, void *kpool, void *vpool,
                           const int32_t *block_table, const int32_t *L0, int32_t num_pages, int32_t page_size,
                           int32_t max_pages, int32_t max_len, int32_t dtype, cudaStream_t stream) {
    ikvgen_spec s = *spec;
    int64_t per_row = (int64_t)max_len * s.head_dim;
    int gx = (int)((per_row + 255) / 256);
    if (gx > 4096) gx = 4096;
    if (gx < 1) gx = 1;
    dim3 grid(gx, s.layers * s.kv_heads, s.batch);
    if (dtype == IKVGEN_BF16)
        fill_paged_kernel<IKVGEN_BF16><<<grid, 256, 0, stream>>>(s, u, kpool, vpool, block_table, L0, num_pages,
                                                                 page_size, max_pages, max_len);
    else
        fill_paged_kernel<IKVGEN_F32><<<grid, 256, 0, stream>>>(s, u, kpool, vpool, block_table, L0, num_pages,
                                                                page_size, max_pages, max_len);
    return (int)cudaGetLastError();
}

int ikvgen_fill_tokens_cuda(const ikvgen_spec *spec, const float *u, const int32_t *L0, int32_t t0, int32_t t1,
                            int32_t dtype, void *out_k, void *out_v, cudaStream_t stream) {
    ikvgen_spec s = *spec;
    int64_t n = (int64_t)(t1 - t0) * s.layers * s.batch * s.kv_heads * s.head_dim;
    int gx = (int)((n + 255) / 256);
    if (gx > 65536) gx = 65536;
    if (gx < 1) gx = 1;
    if (dtype == IKVGEN_BF16)
        fill_tokens_kernel<IKVGEN_BF16><<<gx, 256, 0, stream>>>(s, u, L0, t0, t1, out_k, out_v);
    else
        fill_tokens_kernel<IKVGEN_F32><<<gx, 256, 0, stream>>>(s, u, L0, t0, t1, out_k, out_v);
    return (int)cudaGetLastError();
}

int ikvgen_normals_cuda(uint64_t seed, uint64_t stream_id, int64_t n, float *out, cudaStream_t stream) {
    int gx = (int)((n + 255) / 256);
    if (gx > 65536) gx = 65536;
    if (gx < 1) gx = 1;
    normals_kernel<<<gx, 256, 0, stream>>>(seed, stream_id, n, out);
    return (int)cudaGetLastError();
}

}  // extern "C"
