// Budgeted selection: keep the B highest utilities of a row (Sec. 3: evict the
// lowest m whenever the cache exceeds B).
//
// One 1024-thread CTA per utility row.  Utilities map to order-preserving
// 32-bit keys (sign-flipped IEEE bits; -0.0 folded onto +0.0; NaN -> 1, below
// every number).  Dead slots (pos < 0, deferred compaction) get key 0: below
// every live key, never kept, not counted against B.  General case: an
// MSB-first radix select with 8-bit digits (four passes, warp-aggregated
// shared-memory histograms) finds the exact B-th largest key theta and how
// many theta-valued slots survive; one more pass writes the kept slots in
// ascending order (two block scans per 1024-slot chunk), keeping the lowest
// slots among keys equal to theta.  Steady-state case, one live slot too many:
// a single pass finds the slot to evict (lowest key, and among equal keys the
// highest slot).  The result depends only on the fp32 values, so it is
// bit-exact against any correct sort.
#include "select_row.cuh"

namespace ikv {
namespace {

__global__ void __launch_bounds__(kSelThreads) select_kernel(int32_t cap, const float *__restrict__ util,
                                                              const int32_t *__restrict__ len, int32_t rps,
                                                              const int32_t *__restrict__ budget, int32_t *pos,
                                                              int32_t *keep, int32_t *keep_len, DeferArgs df) {
    pdl_wait();
    select_row(blockIdx.x, cap, util, len, rps, budget, pos, keep, keep_len, df);
}

}  // namespace

cudaError_t launch_select(int32_t rows, int32_t cap, const float *util, const int32_t *len, int32_t rows_per_seq,
                          const int32_t *budget, int32_t *pos, int32_t *keep, int32_t *keep_len, const DeferArgs &df,
                          cudaStream_t st) {
    if (rows <= 0) return cudaSuccess;
    cudaError_t e = launch_k(select_kernel, dim3(rows), dim3(kSelThreads), 0, st, cap, util, len, rows_per_seq, budget,
                             pos, keep, keep_len, df);
    if (e != cudaSuccess) return e;
    note_launch();
    return cudaGetLastError();
}

}  // namespace ikv
