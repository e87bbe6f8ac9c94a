// In-place gather compaction of the paged K/V after eviction, and the append
// of each step's new token.
//
// Stable mode: logical slot j <- logical slot keep[j] for j < n; keep ascending,
// so keep[j] >= j and once keep[j] != j every later slot moves too: only the
// suffix from the first moved slot is touched.  One CTA per (sequence, layer,
// kv head) walks that suffix in ascending 32-row tiles through a 4-stage
// cp.async ring.  A tile's sources are >= its first destination, and every
// earlier tile's destinations lie below that, so reading ahead of the writes is
// safe; within a tile all reads land (wait + barrier) before any write.
// Shorter-side stable mode: with D = len - n evictions, keep[j] - j rises from 0
// to at most D, so either the suffix moves left (start kept) or the prefix before
// the first slot with keep[j] = j + D moves right by its gap (start += D) --
// whichever moves fewer rows.  The right move walks descending tiles, the mirror
// image of the left one.  start only grows that way, so when the right move
// finds no room for the next append before cap, every row moves to slot 0 once
// (an ascending left move with start = 0), provided that frees at least 128
// slots of room; otherwise the suffix moves left.  Survivors keep their order
// in every case.  Extra CTAs per row gather the utility and position arrays
// (logical slots, always left).
//
// Hole-fill mode: survivors at slots >= n move into the evicted slots below n
// (k-th hole <- k-th such survivor).  Sources and destinations are disjoint,
// so every move is independent; the move list is built per row first.
#include "ikv_internal.cuh"

namespace ikv {
namespace {

constexpr int kCompThreads = 256;
constexpr int kCompRows = 32;
constexpr int kRelocateSlack = 128;  // slots a relocation to slot 0 must free
constexpr int kCompStages = 4;

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem) {
    const uint32_t s = static_cast<uint32_t>(__cvta_generic_to_shared(smem));
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

__device__ __forceinline__ int block_min_int(int v, int *scratch) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
    if ((threadIdx.x & 31) == 0) scratch[threadIdx.x >> 5] = v;
    __syncthreads();
    int r = scratch[0];
    for (int w = 1; w < (int)(blockDim.x >> 5); ++w) r = min(r, scratch[w]);
    __syncthreads();
    return r;
}

__device__ __forceinline__ float block_sum(float v, float *scratch) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if ((threadIdx.x & 31) == 0) scratch[threadIdx.x >> 5] = v;
    __syncthreads();
    float r = 0.f;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) r += scratch[w];
    __syncthreads();
    return r;
}

// Logical gather of one per-slot row in place: row[j] <- row[kp[j]] for j < n (kp
// ascending, kp[j] >= j).  Chunk by chunk, every read lands before any write; a
// later chunk's sources lie at or after its own slots, above every earlier write.
template <typename T>
__device__ __forceinline__ void gather_row(T *row, const int32_t *kp, int n) {
    constexpr int PER = 16;
    for (int base = 0; base < n; base += kCompThreads * PER) {
        T val[PER];
        int src[PER];
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int j = base + u * kCompThreads + (int)threadIdx.x;
            src[u] = j < n ? kp[j] : j;
            if (j < n && src[u] != j) val[u] = row[src[u]];
        }
        __syncthreads();
#pragma unroll
        for (int u = 0; u < PER; ++u) {
            const int j = base + u * kCompThreads + (int)threadIdx.x;
            if (j < n && src[u] != j) row[j] = val[u];
        }
        __syncthreads();
    }
}

// Deferred compaction: sequence b only marks its evicted slots dead while its dead
// slots (the ones already dead plus this step's evictions: len - kept) stay within
// max_holes.  Every row of b keeps the same number of slots, so row b * rps decides.
// A sequence whose slot space has no room left for the next append (start + len
// = cap) compacts instead.
__device__ __forceinline__ bool defer_of(const CompactArgs &a, int b, int L, int S) {
    return a.max_holes > 0 && L - a.keep_len[b * a.rows_per_seq] <= a.max_holes && S + L < a.cap;
}

// pos = -1 at every slot below L of row r that keep[r] does not list (runs of
// slots between consecutive kept slots; keep is ascending).
__device__ __forceinline__ void mark_dead_row(const CompactArgs &a, int r, int L) {
    const int n = a.keep_len[r];
    const int32_t *kp = a.keep + (int64_t)r * a.cap;
    int32_t *pos = a.pos + (int64_t)r * a.cap;
    for (int i = threadIdx.x; i <= n; i += blockDim.x) {
        const int lo = i == 0 ? 0 : kp[i - 1] + 1;
        const int hi = i == n ? L : kp[i];
        for (int j = lo; j < hi; ++j) pos[j] = -1;
    }
}

// Stable compaction of one item of sequence b (see the file comment): item x < nkv moves
// the K/V rows of (layer, KV head) x, item nkv + rr gathers utility / position row rr.
// Every item of b reads len[b] and start[b] first; the last of b's items to arrive
// writes the new values, so no item sees them early.  Entered by every thread of the CTA.
__device__ __forceinline__ void compact_stable_item(const CompactArgs &a, const int x, const int b,
                                                    unsigned char *cbuf, int *scratch) {
    const int tid = threadIdx.x;
    const int kvh = a.pv.kv_heads;
    const int nkv = a.layers * kvh;
    if (a.keep_len[b * a.rows_per_seq] < 0) return;  // selection marked the victim dead: nothing to do
    const int L = a.len[b];
    const int S = a.start ? a.start[b] : 0;
    if (defer_of(a, b, L, S)) {  // nothing moves; len, start and the arrival counter stay as they are
        if (x >= nkv) mark_dead_row(a, b * a.rows_per_seq + (x - nkv), L);
        return;
    }
    // shorter-side decision, identical in every CTA of b (it depends on row b only;
    // rows of several KV heads share b's slot space, so they always compact left).
    // K/V row j lands at physical slot new_start + j; it moves iff S + kp[j] differs.
    int new_start = S;
    const int r0 = b * a.rows_per_seq;
    const int n0 = a.keep_len[r0];
    const int32_t *kp0 = a.keep + (int64_t)r0 * a.cap;
    if (a.mode == IKV_COMPACT_STABLE_SHORT && a.rows_per_seq == 1 && a.start && n0 < L) {
        const int D = L - n0;  // evicted slots: the prefix may shift right by D
        int jl = n0, jr = n0;
        for (int j = tid; j < n0; j += kCompThreads) {
            const int kj = kp0[j];
            if (kj != j) jl = min(jl, j);          // left: the suffix from jl moves
            if (kj - j == D) jr = min(jr, j);      // right: the prefix before jr moves
        }
        jl = block_min_int(jl, scratch);
        jr = block_min_int(jr, scratch);
        // room for the appends until the next compaction: one, plus max_holes deferred ones
        const int need = n0 + 1 + max(a.max_holes, 0);
        if (jr < n0 - jl) {
            if (S + D + need <= a.cap)                              // the prefix moves right
                new_start = S + D;
            else if (S > 0 && a.cap - need >= kRelocateSlack)       // out of room: move all rows
                new_start = 0;                                      // to slot 0 once, regaining it
        }
    }
    // whatever the mode, the next append must find a free slot: else move every row to slot 0
    if (a.start && new_start + n0 + 1 > a.cap) new_start = 0;
    if (x < nkv) {
        const int l = x / kvh, g = x % kvh;
        const int r = b * a.rows_per_seq + (a.row_by_layer ? l : a.rows_per_seq == 1 ? 0 : g);
        const int n = a.keep_len[r];
        const int32_t *kp = a.keep + (int64_t)r * a.cap;
        const int shift = new_start - S;
        // right (shift > 0): rows [0, j1) move, j1 the first row already in place (kp[j] = j + shift);
        // left (shift <= 0): rows [j0, n) move, j0 the first row not in place
        const bool right = shift > 0;
        int first = n;
        for (int j = tid; j < n; j += kCompThreads)
            if ((kp[j] == j + shift) == right) first = min(first, j);
        first = block_min_int(first, scratch);
        const int j0 = right ? 0 : first, j1 = right ? first : n;
        if (j0 < j1) {
            const int rowB = a.pv.head_dim * a.elem_bytes;
            const int CPR = rowB >> 4;
            const int stageB = 2 * kCompRows * rowB;
            const int n_tiles = (j1 - j0 + kCompRows - 1) / kCompRows;
            unsigned char *kb = reinterpret_cast<unsigned char *>(a.k);
            unsigned char *vb = reinterpret_cast<unsigned char *>(a.v);
            // tile k covers rows [jb, jb + kCompRows) ascending (left) or descending (right)
            auto tile_base = [&](int tile) { return right ? j1 - (tile + 1) * kCompRows : j0 + tile * kCompRows; };
            auto issue = [&](int tile) {
                unsigned char *st = cbuf + (tile % kCompStages) * stageB;
                const int jb = tile_base(tile);
                for (int idx = tid; idx < kCompRows * CPR; idx += kCompThreads) {
                    const int jj = idx / CPR, c = idx % CPR;
                    const int j = jb + jj;
                    if (j >= j0 && j < j1) {
                        const int64_t src = a.pv.row_phys(b, l, g, S + kp[j]);
                        cp_async16(st + jj * rowB + c * 16, kb + src * rowB + c * 16);
                        cp_async16(st + (kCompRows + jj) * rowB + c * 16, vb + src * rowB + c * 16);
                    }
                }
            };
#pragma unroll
            for (int i = 0; i < kCompStages - 1; ++i) {
                if (i < n_tiles) issue(i);
                cp_async_commit();
            }
            for (int tile = 0; tile < n_tiles; ++tile) {
                __syncthreads();  // the stage about to be refilled was written out last iteration
                if (tile + kCompStages - 1 < n_tiles) issue(tile + kCompStages - 1);
                cp_async_commit();
                cp_async_wait<kCompStages - 1>();
                __syncthreads();  // every read of this tile has landed before any write
                const unsigned char *st = cbuf + (tile % kCompStages) * stageB;
                const int jb = tile_base(tile);
                for (int idx = tid; idx < kCompRows * CPR; idx += kCompThreads) {
                    const int jj = idx / CPR, c = idx % CPR;
                    const int j = jb + jj;
                    if (j >= j0 && j < j1) {
                        const int64_t dst = a.pv.row_phys(b, l, g, new_start + j);
                        *reinterpret_cast<uint4 *>(kb + dst * rowB + c * 16) =
                            *reinterpret_cast<const uint4 *>(st + jj * rowB + c * 16);
                        *reinterpret_cast<uint4 *>(vb + dst * rowB + c * 16) =
                            *reinterpret_cast<const uint4 *>(st + (kCompRows + jj) * rowB + c * 16);
                    }
                }
            }
            cp_async_wait<0>();
        }
        if (a.vnorm) gather_row(a.vnorm + (((int64_t)l * a.batch + b) * kvh + g) * a.cap, kp, n);
    } else {
        // utility / position rows: always the plain stable gather of logical slots
        const int rr = x - nkv;
        const int r = b * a.rows_per_seq + rr;
        const int n = a.keep_len[r];
        const int32_t *kp = a.keep + (int64_t)r * a.cap;
        int32_t *pos = a.pos + (int64_t)r * a.cap;
        float *ema = a.ema ? a.ema + (int64_t)r * a.cap : nullptr;
        constexpr int PER = 16;
        for (int base = 0; base < n; base += kCompThreads * PER) {
            int32_t pv[PER];
            float ev[PER];
            int src[PER];
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                const int j = base + u * kCompThreads + tid;
                src[u] = j < n ? kp[j] : j;
                if (j < n && src[u] != j) {
                    pv[u] = pos[src[u]];
                    ev[u] = ema ? ema[src[u]] : 0.f;
                }
            }
            __syncthreads();
#pragma unroll
            for (int u = 0; u < PER; ++u) {
                const int j = base + u * kCompThreads + tid;
                if (j < n && src[u] != j) {
                    pos[j] = pv[u];
                    if (ema) ema[j] = ev[u];
                }
            }
            __syncthreads();
        }
    }
    // publish len / start once every item of b has read them
    __syncthreads();
    if (tid == 0) {
        if (arrive_acq_rel(&a.done[b]) == nkv + a.rows_per_seq - 1) {
            a.len[b] = n0;
            if (a.start) a.start[b] = new_start;
            a.done[b] = 0;
        }
    }
}

// The stable compaction, one CTA per item: grid (items per sequence, sequences).
__global__ void __launch_bounds__(kCompThreads) compact_stable_kernel(const CompactArgs a) {
    pdl_wait();
    extern __shared__ __align__(16) unsigned char cbuf[];
    __shared__ int scratch[32];
    compact_stable_item(a, blockIdx.x, blockIdx.y, cbuf, scratch);
}

// The same over a fixed grid of one wave of CTAs, for launches with more items than fit
// at once: CTA i takes items i, i + gridDim.x, ... of the (sequence, item) list.  Items of
// a sequence whose row the selection flagged (keep_len < 0: the victim is marked dead,
// nothing moves) are skipped; their flags are read for 32 of the CTA's items at once, so a
// step in which nothing moves costs one round of loads per CTA.  (One CTA per item: 16
// sequences x 257 items of 64 KB shared memory took ~9 launch waves just to exit.)
__global__ void __launch_bounds__(kCompThreads) compact_stable_strided_kernel(const CompactArgs a) {
    pdl_wait();
    extern __shared__ __align__(16) unsigned char cbuf[];
    __shared__ int scratch[32];
    __shared__ int flagged[32];
    const int nx = a.layers * a.pv.kv_heads + a.rows_per_seq;
    const int n_items = nx * a.batch;
#pragma unroll 1
    for (int k0 = 0; blockIdx.x + (int64_t)k0 * gridDim.x < n_items; k0 += 32) {
        if (threadIdx.x < 32) {
            const int64_t item = blockIdx.x + (int64_t)(k0 + threadIdx.x) * gridDim.x;
            flagged[threadIdx.x] = item < n_items ? a.keep_len[(int)(item / nx) * a.rows_per_seq] < 0 : 1;
        }
        __syncthreads();
#pragma unroll 1
        for (int k = 0; k < 32; ++k) {
            const int64_t item = blockIdx.x + (int64_t)(k0 + k) * gridDim.x;
            if (item >= n_items) break;
            if (flagged[k]) continue;
            compact_stable_item(a, (int)(item % nx), (int)(item / nx), cbuf, scratch);
            __syncthreads();  // the next item reuses the shared buffers
        }
        __syncthreads();  // flagged is rewritten
    }
}

// Hole-fill move list of one row: for every evicted slot h < n (the k-th such),
// move the k-th survivor found at a slot >= n into it.  keep is ascending, so the
// gap g_j = keep[j] - j is non-decreasing over the `below` survivors < n; the
// holes just before keep[j] are the g_j - g_{j-1} slots keep[j] - g_j + k for
// hole indices k in [g_{j-1}, g_j), and the holes after the last of them are the
// slots below + k.  One coalesced pass over keep, no searching.
constexpr int kPlanThreads = 1024;

__global__ void __launch_bounds__(kPlanThreads) holefill_plan_kernel(const CompactArgs a) {
    pdl_wait();
    __shared__ int below_s;
    const int r = blockIdx.x;
    const int n = a.keep_len[r];
    if (n < 0) return;  // selection marked the victim dead: nothing to do
    const int32_t *kp = a.keep + (int64_t)r * a.cap;
    if (defer_of(a, r / a.rows_per_seq, a.len[r / a.rows_per_seq], a.pv.start_of(r / a.rows_per_seq))) {
        // decided here, before len changes
        if (threadIdx.x == 0) a.n_moves[r] = -1;
        return;
    }
    if (threadIdx.x == 0) below_s = 0;
    __syncthreads();
    int cnt = 0;
    for (int j = threadIdx.x; j < n; j += kPlanThreads) cnt += kp[j] < n;
    if (cnt) atomicAdd(&below_s, cnt);
    __syncthreads();
    const int below = below_s;       // survivors already below n
    const int n_tail = n - below;    // survivors at slots >= n = holes below n
    int32_t *mv = a.moves + (int64_t)r * a.cap * 2;
    for (int j = threadIdx.x; j < below; j += kPlanThreads) {
        const int kj = kp[j];
        const int g = kj - j, gp = j ? kp[j - 1] - (j - 1) : 0;
        for (int k = gp; k < g; ++k) {
            mv[2 * k] = kp[below + k];
            mv[2 * k + 1] = kj - g + k;
        }
    }
    const int g_last = below ? kp[below - 1] - (below - 1) : 0;
    for (int k = g_last + threadIdx.x; k < n_tail; k += kPlanThreads) {
        mv[2 * k] = kp[below + k];
        mv[2 * k + 1] = below + k;
    }
    if (threadIdx.x == 0) a.n_moves[r] = n_tail;
}

__global__ void __launch_bounds__(kCompThreads) holefill_move_kernel(const CompactArgs a) {
    pdl_wait();
    const int tid = threadIdx.x;
    const int b = blockIdx.y, x = blockIdx.x;
    const int kvh = a.pv.kv_heads;
    const int nkv = a.layers * kvh;
    if (a.keep_len[b * a.rows_per_seq] < 0) return;  // selection marked the victim dead: nothing to do
    if (x < nkv) {
        const int l = x / kvh, g = x % kvh;
        const int r = b * a.rows_per_seq + (a.row_by_layer ? l : a.rows_per_seq == 1 ? 0 : g);
        const int nm = a.n_moves[r];  // -1: deferred, nothing moves
        const int32_t *mv = a.moves + (int64_t)r * a.cap * 2;
        const int S = a.pv.start_of(b);
        const int rowB = a.pv.head_dim * a.elem_bytes;
        const int CPR = rowB >> 4;
        unsigned char *kb = reinterpret_cast<unsigned char *>(a.k);
        unsigned char *vb = reinterpret_cast<unsigned char *>(a.v);
        if (a.vnorm) {
            float *vn = a.vnorm + (((int64_t)l * a.batch + b) * kvh + g) * a.cap;
            for (int m = tid; m < nm; m += kCompThreads) vn[mv[2 * m + 1]] = vn[mv[2 * m]];
        }
        for (int idx = tid; idx < nm * CPR; idx += kCompThreads) {
            const int m = idx / CPR, c = idx % CPR;
            const int64_t src = a.pv.row_phys(b, l, g, S + mv[2 * m]);
            const int64_t dst = a.pv.row_phys(b, l, g, S + mv[2 * m + 1]);
            *reinterpret_cast<uint4 *>(kb + dst * rowB + c * 16) = *reinterpret_cast<const uint4 *>(kb + src * rowB + c * 16);
            *reinterpret_cast<uint4 *>(vb + dst * rowB + c * 16) = *reinterpret_cast<const uint4 *>(vb + src * rowB + c * 16);
        }
        return;
    }
    const int rr = x - nkv;
    const int r = b * a.rows_per_seq + rr;
    const int nm = a.n_moves[r];
    if (nm < 0) {  // deferred: mark this step's evictions dead; len stays
        mark_dead_row(a, r, a.len[b]);
        return;
    }
    const int32_t *mv = a.moves + (int64_t)r * a.cap * 2;
    int32_t *pos = a.pos + (int64_t)r * a.cap;
    float *ema = a.ema ? a.ema + (int64_t)r * a.cap : nullptr;
    for (int m = tid; m < nm; m += kCompThreads) {
        const int s = mv[2 * m], d = mv[2 * m + 1];
        pos[d] = pos[s];
        if (ema) ema[d] = ema[s];
    }
    if (rr == 0 && tid == 0) a.len[b] = a.keep_len[r];
}

// New token of every sequence into slot len[b] of every layer and kv head.
// CTAs (x, b) copy 8 rows each; CTA 0 also sets the row utilities / positions;
// the last CTA of sequence b to arrive advances len[b] and next_pos[b] (every
// CTA reads len[b] before it arrives, so nobody sees the new value early).
constexpr int kAppendRows = 8;

}  // namespace

__device__ unsigned int g_append_error = 0;  // bit 0: an append found no free slot (start + len = cap)

namespace {

__global__ void __launch_bounds__(kCompThreads) append_kernel(const AppendArgs a) {
    pdl_wait();
    __shared__ float scratch[32];
    const int tid = threadIdx.x;
    const int b = blockIdx.y;
    const int L = a.len[b];
    const int S = a.pv.start_of(b);
    const int kvh = a.pv.kv_heads;
    const int nkv = a.layers * kvh;
    const int rowB = a.pv.head_dim * a.elem_bytes;
    const int CPR = rowB >> 4;
    if (a.slot && blockIdx.x == 0 && tid == 0) a.slot[b] = S + L < a.cap ? L : -1;
    if (S + L < a.cap && a.k_new) {
        unsigned char *kb = reinterpret_cast<unsigned char *>(a.k);
        unsigned char *vb = reinterpret_cast<unsigned char *>(a.v);
        const unsigned char *kn = reinterpret_cast<const unsigned char *>(a.k_new);
        const unsigned char *vn = reinterpret_cast<const unsigned char *>(a.v_new);
        for (int idx = tid; idx < kAppendRows * CPR; idx += kCompThreads) {
            const int x = blockIdx.x * kAppendRows + idx / CPR, c = idx % CPR;
            if (x < nkv) {
                const int l = x / kvh, g = x % kvh;
                const int64_t src = (((int64_t)l * a.batch + b) * kvh + g) * rowB + c * 16;
                const int64_t dst = a.pv.row_phys(b, l, g, S + L) * rowB + c * 16;
                *reinterpret_cast<uint4 *>(kb + dst) = *reinterpret_cast<const uint4 *>(kn + src);
                *reinterpret_cast<uint4 *>(vb + dst) = *reinterpret_cast<const uint4 *>(vn + src);
            }
        }
        if (a.vnorm) {  // l2 norm of the new value row: warp w takes the CTA's row w
            const int x = blockIdx.x * kAppendRows + (tid >> 5), lane = tid & 31;
            if ((tid >> 5) < kAppendRows && x < nkv) {
                const int l = x / kvh, g = x % kvh;
                const int64_t e0 = (((int64_t)l * a.batch + b) * kvh + g) * a.pv.head_dim;
                float sq = 0.f;
                for (int e = lane; e < a.pv.head_dim; e += 32) {
                    const float xv = a.elem_bytes == 2
                                         ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.v_new)[e0 + e])
                                         : reinterpret_cast<const float *>(a.v_new)[e0 + e];
                    sq += xv * xv;
                }
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
                if (lane == 0) a.vnorm[(((int64_t)l * a.batch + b) * kvh + g) * a.cap + L] = sqrtf(sq);
            }
        }
    }
    if (S + L < a.cap) {
        if (blockIdx.x == 0) {
            const int np = a.next_pos[b];
            for (int rr = 0; rr < a.rows_per_seq; ++rr) {
                const int64_t r = (int64_t)b * a.rows_per_seq + rr;
                float init = 0.f;
                if (a.init_mean && L > 0) {
                    float s = 0.f, c = 0.f;
                    const int32_t *pr = a.pos + r * a.cap;
                    for (int i = tid; i < L; i += kCompThreads)
                        if (!a.dead_slots || pr[i] >= 0) {  // the mean over live slots only
                            s += a.ema[r * a.cap + i];
                            c += 1.f;
                        }
                    s = block_sum(s, scratch);
                    c = a.dead_slots ? block_sum(c, scratch) : (float)L;
                    init = c > 0.f ? s / c : 0.f;
                }
                if (tid == 0) {
                    if (a.ema) a.ema[r * a.cap + L] = init;
                    a.pos[r * a.cap + L] = np;
                }
            }
        }
    }
    __syncthreads();
    if (gridDim.x == 1) {
        // bookkeeping only (one CTA per sequence, which has read len[b] above): no arrival
        if (tid == 0) {
            if (S + L < a.cap) {
                a.len[b] = L + 1;
                a.next_pos[b] = a.next_pos[b] + 1;
            } else {
                atomicOr(&g_append_error, 1u);  // the token was not stored; ikv_device_status reports it
            }
        }
        return;
    }
    if (tid == 0) {
        if (arrive_acq_rel(&a.done[b]) == (int)gridDim.x - 1) {
            if (S + L < a.cap) {
                a.len[b] = L + 1;
                a.next_pos[b] = a.next_pos[b] + 1;
            } else {
                atomicOr(&g_append_error, 1u);  // the token was not stored; ikv_device_status reports it
            }
            a.done[b] = 0;
        }
    }
}

// Split step: the new token's rows of layers layer0 .. layer0 + layers - 1 into the
// slot the begin call reserved.  CTA (x, b) copies (layer, kv head) rows 8x .. 8x+7 of
// sequence b and stores their value-row norms.
__global__ void __launch_bounds__(kCompThreads) append_rows_kernel(const AppendArgs a) {
    pdl_wait();
    const int tid = threadIdx.x;
    const int b = blockIdx.y;
    const int kvh = a.pv.kv_heads;
    const int nkv = a.layers * kvh;
    const int j = a.slot[b];
    if (j < 0) return;  // no room: the begin call flagged the error and kept len
    const int S = a.pv.start_of(b);
    const int rowB = a.pv.head_dim * a.elem_bytes;
    const int CPR = rowB >> 4;
    unsigned char *kb = reinterpret_cast<unsigned char *>(a.k);
    unsigned char *vb = reinterpret_cast<unsigned char *>(a.v);
    const unsigned char *kn = reinterpret_cast<const unsigned char *>(a.k_new);
    const unsigned char *vn = reinterpret_cast<const unsigned char *>(a.v_new);
    for (int idx = tid; idx < kAppendRows * CPR; idx += kCompThreads) {
        const int x = blockIdx.x * kAppendRows + idx / CPR, c = idx % CPR;
        if (x < nkv) {
            const int li = x / kvh, g = x % kvh;
            const int64_t src = (((int64_t)li * a.batch + b) * kvh + g) * rowB + c * 16;
            const int64_t dst = a.pv.row_phys(b, a.layer0 + li, g, S + j) * rowB + c * 16;
            *reinterpret_cast<uint4 *>(kb + dst) = *reinterpret_cast<const uint4 *>(kn + src);
            *reinterpret_cast<uint4 *>(vb + dst) = *reinterpret_cast<const uint4 *>(vn + src);
        }
    }
    if (a.vnorm) {
        const int x = blockIdx.x * kAppendRows + (tid >> 5), lane = tid & 31;
        if ((tid >> 5) < kAppendRows && x < nkv) {
            const int li = x / kvh, g = x % kvh;
            const int64_t e0 = (((int64_t)li * a.batch + b) * kvh + g) * a.pv.head_dim;
            float sq = 0.f;
            for (int e = lane; e < a.pv.head_dim; e += 32) {
                const float xv = a.elem_bytes == 2
                                     ? __bfloat162float(reinterpret_cast<const __nv_bfloat16 *>(a.v_new)[e0 + e])
                                     : reinterpret_cast<const float *>(a.v_new)[e0 + e];
                sq += xv * xv;
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
            if (lane == 0) a.vnorm[(((int64_t)(a.layer0 + li) * a.batch + b) * kvh + g) * a.cap + j] = sqrtf(sq);
        }
    }
}

}  // namespace

cudaError_t launch_compact(const CompactArgs &a, int mode, int sms, cudaStream_t st) {
    dim3 grid(a.layers * a.pv.kv_heads + a.rows_per_seq, a.batch);
    if (mode == IKV_COMPACT_STABLE || mode == IKV_COMPACT_STABLE_SHORT) {
        const int smem = kCompStages * 2 * kCompRows * a.pv.head_dim * a.elem_bytes;
        static int attr_smem = 0;  // raise the dynamic shared-memory limits once per size
        static int per_sm = 0;     // resident CTAs per SM of the strided kernel at attr_smem
        if (smem > attr_smem || per_sm == 0) {
            cudaError_t e =
                cudaFuncSetAttribute(compact_stable_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
            if (e == cudaSuccess)
                e = cudaFuncSetAttribute(compact_stable_strided_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         smem);
            if (e == cudaSuccess)
                e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, compact_stable_strided_kernel,
                                                                  kCompThreads, smem);
            if (e != cudaSuccess) return e;
            if (per_sm < 1) per_sm = 1;
            attr_smem = smem;
        }
        const int64_t items = (int64_t)grid.x * grid.y;
        const int64_t wave = (int64_t)per_sm * (sms > 0 ? sms : 1);
        cudaError_t e = items <= wave
                            ? launch_k(compact_stable_kernel, grid, dim3(kCompThreads), smem, st, a)
                            : launch_k(compact_stable_strided_kernel, dim3((unsigned)wave), dim3(kCompThreads), smem,
                                       st, a);
        note_launch();
        return e != cudaSuccess ? e : cudaGetLastError();
    }
    cudaError_t e = launch_k(holefill_plan_kernel, dim3(a.batch * a.rows_per_seq), dim3(kPlanThreads), 0, st, a);
    note_launch();
    if (e != cudaSuccess) return e;
    e = launch_k(holefill_move_kernel, grid, dim3(kCompThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t read_clear_append_error(unsigned int *v) {
    unsigned int z = 0;
    cudaError_t e = cudaMemcpyFromSymbol(v, g_append_error, sizeof(*v));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(g_append_error, &z, sizeof(z));
    return e;
}

cudaError_t launch_append(const AppendArgs &a, cudaStream_t st) {
    const int nkv = a.layers * a.pv.kv_heads;
    dim3 grid(a.k_new ? (nkv + kAppendRows - 1) / kAppendRows : 1, a.batch);
    cudaError_t e = launch_k(append_kernel, grid, dim3(kCompThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_append_rows(const AppendArgs &a, cudaStream_t st) {
    dim3 grid((a.layers * a.pv.kv_heads + kAppendRows - 1) / kAppendRows, a.batch);
    cudaError_t e = launch_k(append_rows_kernel, grid, dim3(kCompThreads), 0, st, a);
    note_launch();
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace ikv
