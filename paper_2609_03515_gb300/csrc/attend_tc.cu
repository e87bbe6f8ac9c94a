// Tensor-core split-K decode attention with logits, bf16, head_dim 128 (sm_103a).
//
// The cache of every (sequence, layer, kv head) unit is cut into chunks of up to
// 15 tiles of 128 tokens; one CTA handles one chunk, or several consecutive
// chunks as passes (the G query heads of its kv head), writes their log2-domain
// logits and its (max, sum, O) partial, and the unit's last CTA to finish merges
// the partials into the output and the per-head log-sum-exp (arrival counter, no
// waiting); a unit covered by one CTA writes them directly.  The 1-D grid is
// chunk-major, so every unit's short remainder chunk is dispatched last and fills
// the final wave.  Two CTAs share an SM.  Built from Blackwell pieces:
//   * TMA (cp.async.bulk.tensor.2d, 128-byte swizzle) streams 128-token K and V
//     tiles out of the paged pool (one box per page segment and 64-column half)
//     into a 3-stage ring guarded by mbarriers;
//   * tcgen05.mma (kind::f16, bf16 in, fp32 accumulate in TMEM) computes
//       S_i[128 tokens x 16] = K_i[128 x 128] . Q^T[128 x 16]   (Q: G heads, zero-padded to 16)
//       O[128 dims x 16]    += V_i^T[128 x 128] . P_i^T[128 x 16]
//     with K-major operands for QK and an MN-major (transposed) V for PV;
//   * the softmax runs as two sweeps over the S tiles kept in TMEM: the chunk
//     maximum per head, then logits write-out, exp2, row sums and the bf16 P
//     operand (double-buffered in shared memory) that feeds the PV MMA;
//   * between passes the softmax frees the S tiles and O (s_free, o_free
//     barriers) and folds the pass's (max, sum, O) into running registers, the
//     online-softmax rescaling by exp2(m_old - m_new).
// Warp roles (192 threads): warps 0-3 own TMEM lanes 0-127 (softmax, epilogue),
// warp 4 issues TMA loads, warp 5 issues MMAs.  Every mbarrier wait is bounded;
// on timeout the CTA records an error code, stops issuing work, waits for its
// in-flight copies and MMAs, frees its TMEM and returns.
#include <atomic>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "ikv_internal.cuh"

namespace ikv {

__device__ unsigned int g_tc_error = 0;

namespace {

constexpr int kTile = 128;
constexpr int kD = 128;
constexpr int kNst = 3;
constexpr int kStage = kTile * kD * 2;          // 32 KB: one K or V tile
constexpr int kHalf = kStage / 2;               // one 64-column half (16 KB)
constexpr int kN = 16;                          // padded head count (MMA N)
constexpr int kOpBytes = kN * kD * 2;           // 4 KB: Q or one P operand
constexpr int kTmemCols = 256;
constexpr int kOcol = kTmemCols - kN;           // O accumulator columns [240, 256)
constexpr int kMaxTiles = kOcol / kN;           // 15 S tiles
constexpr int kEarlyChunks = 16;                // merge: partial outputs loaded with the (max, sum) pairs
constexpr int kThreads = 192;
constexpr uint64_t kWaitNs = 1000000000ull;   // 1 s: orders of magnitude above any legitimate wait

constexpr int kOffQ = kNst * kStage;
constexpr int kOffP = kOffQ + kOpBytes;
constexpr int kOffRed = kOffP + 2 * kOpBytes;
constexpr int kOffNew = kOffRed + 4 * kN * 4;   // split step: the new token's K and V rows (2 x 256 B)
constexpr int kOffBar = kOffNew + 2 * kD * 2;
// barriers: full[kNst], empty[kNst], s_full, p_full[2], p_empty[2], o_full, s_free, o_free, mma_done,
// stall (the bounded-wait test's barrier, which nothing arrives at)
constexpr int kNumBar = 2 * kNst + 10;
constexpr uint64_t kStallNs = 10000ull;       // the bounded-wait test's limit: 10 us
constexpr int kOffMisc = kOffBar + kNumBar * 8;
constexpr int kSmemBytes = kOffMisc + 16 + 1024;  // misc: tmem slot, abort flag, last-split flag   // + slack for 1024-byte alignment

enum : unsigned { kErrTimeout = 1u };

struct TcArgs {
    const int32_t *len;
    const int32_t *block_table;
    const int32_t *start;       // [batch] physical slot of logical slot 0, or null
    int32_t num_pages, page_size, max_pages, kv_heads, rows_per_box;
    const __nv_bfloat16 *q;     // q + ((li*batch + b)*H + h)*128
    int32_t batch, q_heads, layer0, n_layers, split_tokens, n_splits, cap;
    float scale_log2;
    float *logits;              // may be null; [batch][sc_layers][H][lstride]
    int32_t lstride;            // logits row stride, a multiple of 128
    float *part_ml, *part_o;
    __nv_bfloat16 *out;         // [n_layers][batch][H][128]
    float *lse2;                // [batch][sc_layers][H]
    int32_t *arrivals;          // [batch][n_layers][kv_heads], zero on entry, left zero
    const int32_t *pos;         // [rows][cap], -1 at dead slots; null: every slot below len is live
    int32_t rows_per_seq;
    int32_t sc_layers, sc_layer0;  // local layer li is layer sc_layer0 + li of logits / lse2
    // the new token's K/V rows ([n_layers][batch][kv_heads][128]) go to logical slot slot[b]
    // (-1: none), written by the CTA whose chunk holds it, which also uses them in place of
    // the slot's old contents; vnorm (or null) gets their V norms
    const __nv_bfloat16 *k_new, *v_new;
    const int32_t *slot;
    __nv_bfloat16 *k_pool, *v_pool;
    float *vnorm;
    // every unit is a single chunk: instead of per-head logits, write per token the KV
    // head's group sum of normalised probabilities, [batch][sc_layers][kv_heads][lstride]
    int32_t gsum;
    int32_t passes;  // consecutive chunks per CTA (>= 1)
    // nonzero: nothing the preceding kernels in the stream still write is read before the
    // programmatic-dependency wait except through this launch's own new-token rows, so the
    // CTA initialises and starts streaming its K/V tiles first (a later layer call of the
    // split step: len, start, slot, pos, the block table and this layer's cached rows are
    // fixed since the step's first call)
    int32_t early;
    // nonzero (tests of the bounded waits): the MMA issuer first waits, at most kStallNs, on a
    // barrier that nothing arrives at, so the wait runs out and the CTA takes its abort path
    int32_t stall;
};

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Bounded wait on an mbarrier phase (non-blocking polls, at most kWaitNs of wall
// time).  Returns false -- raising the CTA's abort flag and the global error
// word -- if the phase does not complete in time, or returns false at once if
// another role of the CTA has already aborted.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort,
                                          uint64_t limit_ns = kWaitNs) {
    if (mbar_test(bar, parity)) return true;
    const uint64_t start = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_test(bar, parity)) return true;
        if (i > 64) __nanosleep(32);
        if ((i & 63u) == 0) {
            if (*abort) return false;
            if (global_ns() - start > limit_ns) break;
        }
    }
    *abort = 1;
    atomicOr(&g_tc_error, kErrTimeout);
    return false;
}

// Wait for the MMAs this thread has issued, whatever the abort flag says (at most kWaitNs):
// TMEM is freed only after every tcgen05 operation writing it has completed.
__device__ __forceinline__ void mbar_drain(uint32_t bar, uint32_t parity) {
    const uint64_t start = global_ns();
    for (uint32_t i = 0; !mbar_test(bar, parity); ++i) {
        if (i > 64) __nanosleep(32);
        if ((i & 63u) == 63u && global_ns() - start > kWaitNs) {
            atomicOr(&g_tc_error, kErrTimeout);
            return;
        }
    }
}

// L2 policy for data read once and never again in the step (the K/V stream): its lines are
// the first to go, so the logits this kernel writes for the score pass stay in L2
__device__ __forceinline__ uint64_t l2_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, int x, int y, uint32_t bar,
                                            uint64_t pol) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1, {%2, "
        "%3}], [%4], %5;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar), "l"(pol)
        : "memory");
}

__device__ __forceinline__ void bulk_prefetch_l2(const void *p, uint32_t bytes) {
    asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ void tma_prefetch_2d(const CUtensorMap *map, int x, int y) {
    asm volatile("cp.async.bulk.prefetch.tensor.2d.L2.global [%0, {%1, %2}];" ::"l"(reinterpret_cast<uint64_t>(map)),
                 "r"(x), "r"(y)
                 : "memory");
}

// smem matrix descriptor, 128-byte swizzle (sm_100 family, version 1)
__device__ __forceinline__ uint64_t sdesc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// instruction descriptor kind::f16: bf16 x bf16 -> f32, A K-major or MN-major, B K-major
__host__ __device__ constexpr uint32_t idesc_bf16(bool a_mn_major, int M, int N) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn_major ? 1u : 0u) << 15) | ((uint32_t)(N >> 3) << 17) |
           ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(
            d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void fence_after_sync() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_before_sync() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void fence_async_smem() { asm volatile("fence.proxy.async.shared::cta;" ::: "memory"); }
__device__ __forceinline__ void softmax_bar() { asm volatile("bar.sync 1, 128;" ::: "memory"); }

template <int NC>
__device__ __forceinline__ void tmem_ld(uint32_t taddr, float *v);
template <>
__device__ __forceinline__ void tmem_ld<4>(uint32_t taddr, float *v) {
    uint32_t r[4];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x4.b32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 4; ++i) v[i] = __uint_as_float(r[i]);
}
template <>
__device__ __forceinline__ void tmem_ld<8>(uint32_t taddr, float *v) {
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// byte offset of element (row, col) inside a [rows][64] bf16 block stored with
// the 128-byte swizzle (128-byte rows, 16-byte chunks permuted by row % 8)
__device__ __forceinline__ uint32_t sw128(uint32_t row, uint32_t col) {
    return row * 128u + ((((col >> 3) ^ row) & 7u) << 4) + ((col & 7u) << 1);
}

// MP: the launch may give a CTA more than one pass (a.passes > 1); without it the pass
// loop, the s_free / o_free handshakes and the register fold compile away.
template <int G, bool MP>
__global__ void __launch_bounds__(kThreads, 2)
    attend_tc_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, const TcArgs a) {
    constexpr int NC = G <= 4 ? 4 : 8;  // TMEM columns read per S tile
    const bool early = a.early != 0;
    if (!early) pdl_wait();
    extern __shared__ unsigned char smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    unsigned char *sm = smem_raw + (base - raw);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // 1-D grid, chunk-major: CTA i takes a.passes consecutive chunks of unit i % n_units,
    // starting at chunk (i / n_units) * a.passes, so every unit's short remainder is
    // dispatched last and fills the final wave.  The chunks of one CTA run as passes over
    // the same TMEM columns; their (max, sum, output) are merged in registers.
    const int n_units = a.batch * a.n_layers * a.kv_heads;
    const int cta = blockIdx.x / n_units;  // CTA index within the unit
    const int unit_id = blockIdx.x % n_units;
    const int g = unit_id % a.kv_heads;
    const int b = (unit_id / a.kv_heads) % a.batch, li = (unit_id / a.kv_heads) / a.batch;
    const int l = a.layer0 + li;
    // The unit's valid rows are physical slots [S0, S0 + L).  Chunks cut the 128-aligned
    // physical tiles covering them (TMA boxes stay page aligned); rows outside are masked.
    // (L2 loads: an early CTA reads these before the dependency wait)
    const int L = __ldcg(a.len + b);
    const int S0 = a.start ? __ldcg(a.start + b) : 0;
    const int ft = S0 / kTile;
    const int nt_unit = L > 0 ? (S0 + L + kTile - 1) / kTile - ft : 0;
    const int item = a.split_tokens / kTile;  // tiles per chunk
    const int ns_active = (nt_unit + item - 1) / item;  // chunks of the unit
    const int c0 = cta * a.passes;                      // this CTA's first chunk
    if (c0 >= ns_active) {
        if (early) pdl_wait();
        if (cta == 0) {  // empty sequence: zero output, log-sum-exp -inf
            for (int i = threadIdx.x; i < G * kD; i += kThreads)
                a.out[(((int64_t)li * a.batch + b) * a.q_heads + (int64_t)g * G) * kD + i] = __float2bfloat16_rn(0.f);
            if (threadIdx.x < G)
                a.lse2[((int64_t)b * a.sc_layers + a.sc_layer0 + li) * a.q_heads + (int64_t)g * G + threadIdx.x] =
                    -INFINITY;
        }
        return;
    }
    const int np = MP ? min(a.passes, ns_active - c0) : 1;             // passes of this CTA
    const int nc_unit = MP ? (ns_active + a.passes - 1) / a.passes : ns_active;  // CTAs that cover the unit
    if (item > kMaxTiles) {  // the host sizes chunks to fit TMEM; refuse rather than overrun
        if (threadIdx.x == 0) atomicOr(&g_tc_error, 2u);
        return;
    }
    // pass p: tiles and physical slot of the first row
    auto chunk_n = [&](int p) { return min(item, nt_unit - (c0 + (MP ? p : 0)) * item); };
    auto chunk_t0 = [&](int p) { return (ft + (c0 + (MP ? p : 0)) * item) * kTile; };
    const int H = a.q_heads;

    const uint32_t sQ = base + kOffQ, sP = base + kOffP;
    float *red = reinterpret_cast<float *>(sm + kOffRed);
    const uint32_t bar0 = base + kOffBar;
    auto full = [&](int i) { return bar0 + 8u * i; };
    auto empty = [&](int i) { return bar0 + 8u * (kNst + i); };
    const uint32_t s_full = bar0 + 8u * (2 * kNst);
    auto p_full = [&](int i) { return bar0 + 8u * (2 * kNst + 1 + i); };
    auto p_empty = [&](int i) { return bar0 + 8u * (2 * kNst + 3 + i); };
    const uint32_t o_full = bar0 + 8u * (2 * kNst + 5);
    const uint32_t s_free = bar0 + 8u * (2 * kNst + 6);  // the softmax is done with a pass's S tiles
    const uint32_t o_free = bar0 + 8u * (2 * kNst + 7);  // the softmax has read a pass's O
    const uint32_t mma_done = bar0 + 8u * (2 * kNst + 8);  // every MMA of the CTA has completed
    const uint32_t stall_bar = bar0 + 8u * (2 * kNst + 9);  // nothing arrives here (a.stall)
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(sm + kOffMisc);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(sm + kOffMisc + 4);

    // The load stream: per pass, its K tiles then its V tiles; load J of the stream goes
    // to ring stage J % kNst.  pool row of box bx of load j of pass p:
    const int boxes = kTile / a.rows_per_box;
    auto box_row = [&](int p, int j, int bx) {
        const int n = chunk_n(p);
        const int tile = j < n ? j : j - n;
        const int tok = chunk_t0(p) + tile * kTile + bx * a.rows_per_box;
        int lp = tok / a.page_size;
        if (lp >= a.max_pages) lp = a.max_pages - 1;
        const int page = a.block_table[(int64_t)b * a.max_pages + lp];
        return ((l * a.num_pages + page) * a.kv_heads + g) * a.page_size + tok % a.page_size;
    };
    int ld_J = 0, ld_p = 0, ld_j = 0;  // producer cursor: loads issued, pass and load of the next one
    const uint64_t kv_pol = l2_evict_first();
    // split step: the physical slot that receives the new token's rows (-1: none, or not in
    // this CTA's chunks).  The tiles holding it are loaded like any other; the MMA thread
    // writes the new rows into the loaded K and V tiles before their products read them.
    int p_new = -1;
    if (a.k_new) {
        const int j = __ldcg(a.slot + b);
        const int pn = S0 + j;
        if (j >= 0 && pn >= chunk_t0(0) && pn < chunk_t0(np - 1) + chunk_n(np - 1) * kTile) p_new = pn;
    }
    auto issue_next = [&]() {
        const int st = ld_J % kNst;
        mbar_expect_tx(full(st), kStage);
        const CUtensorMap *tm = ld_j < chunk_n(ld_p) ? &tmK : &tmV;
        const uint32_t dst = base + st * kStage;
        for (int bx = 0; bx < boxes; ++bx) {
            const int row = box_row(ld_p, ld_j, bx);
            tma_load_2d(dst + bx * a.rows_per_box * 128, tm, 0, row, full(st), kv_pol);
            tma_load_2d(dst + kHalf + bx * a.rows_per_box * 128, tm, 64, row, full(st), kv_pol);
        }
        ++ld_J;
        if (++ld_j == 2 * chunk_n(ld_p)) {
            ++ld_p;
            ld_j = 0;
        }
    };
    // Prologue.  The producer lane initialises the barriers and starts the K/V stream at
    // once (every load up to the ring's depth); the TMEM allocation and P zeroing below
    // overlap the loads' latency.  An early CTA does all of this before the dependency
    // wait, so it overlaps the previous kernel's tail.
    if (warp == 4 && lane == 0) {
        for (int i = 0; i < kNst; ++i) {
            mbar_init(full(i), 1);
            mbar_init(empty(i), 1);
        }
        mbar_init(s_full, 1);
        mbar_init(p_full(0), 128);
        mbar_init(p_full(1), 128);
        mbar_init(p_empty(0), 1);
        mbar_init(p_empty(1), 1);
        mbar_init(o_full, 1);
        mbar_init(s_free, 128);
        mbar_init(o_free, 128);
        mbar_init(mma_done, 1);
        mbar_init(stall_bar, 1);
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        while (ld_J < kNst && ld_p < np) issue_next();
        // an early CTA also pulls the rest of its tiles, and its q rows, into L2 while it
        // waits, so the loads it can only issue later find them there (a prefetch cannot
        // return stale data: L2 is where writes land)
        if (early) {
            for (int p = ld_p, j = ld_j; p < np;) {
                const CUtensorMap *tm = j < chunk_n(p) ? &tmK : &tmV;
                for (int bx = 0; bx < boxes; ++bx) {
                    const int row = box_row(p, j, bx);
                    tma_prefetch_2d(tm, 0, row);
                    tma_prefetch_2d(tm, 64, row);
                }
                if (++j == 2 * chunk_n(p)) {
                    ++p;
                    j = 0;
                }
            }
            bulk_prefetch_l2(a.q + (((int64_t)li * a.batch + b) * a.q_heads + (int64_t)g * G) * kD, G * kD * 2);
        }
    }
    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    // both P buffers zeroed (rows >= G stay zero)
    for (int i = tid; i < 2 * kOpBytes / 16; i += kThreads)
        reinterpret_cast<uint4 *>(sm + kOffP)[i] = make_uint4(0, 0, 0, 0);
    if (early) pdl_wait();
    if (warp == 4) {
        // Split step: the CTA whose chunks hold the new token's slot stores the token's K
        // and V rows into the cache (lanes 0-15: K, 16-31: V, 16 bytes each) for later steps,
        // and stages them in shared memory for its own MMAs (the tiles it loads may hold the
        // slot's old contents: the MMA thread overwrites that row before using them)
        if (a.k_new) {
            const int j = p_new - S0;
            const int p = p_new;
            if (p_new >= 0) {
                const int page = a.block_table[(int64_t)b * a.max_pages + p / a.page_size];
                const int64_t row = ((int64_t)(l * a.num_pages + page) * a.kv_heads + g) * a.page_size + p % a.page_size;
                const bool isv = lane >= 16;
                const int c = lane & 15;
                const uint4 x = reinterpret_cast<const uint4 *>(
                    isv ? a.v_new : a.k_new)[(((int64_t)li * a.batch + b) * a.kv_heads + g) * 16 + c];
                reinterpret_cast<uint4 *>(isv ? a.v_pool : a.k_pool)[row * 16 + c] = x;
                reinterpret_cast<uint4 *>(sm + kOffNew)[lane] = x;
                float sq = 0.f;
                if (isv) {
                    const uint32_t w4[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const float lo = __uint_as_float(w4[k] << 16), hi = __uint_as_float(w4[k] & 0xffff0000u);
                        sq += lo * lo + hi * hi;
                    }
                }
#pragma unroll
                for (int o = 8; o > 0; o >>= 1) sq += __shfl_xor_sync(0xffffffffu, sq, o);
                if (a.vnorm && lane == 16)
                    a.vnorm[(((int64_t)l * a.batch + b) * a.kv_heads + g) * a.cap + j] = sqrtf(sq);
            }
            __syncwarp();
        }
    }
    // Q operand [16 heads][128 dims], heads >= G zero: one 16-byte load per thread (8 dims
    // of one head, which stay together as one 16-byte chunk of the swizzled layout)
    {
        const __nv_bfloat16 *qg = a.q + (((int64_t)li * a.batch + b) * H + (int64_t)g * G) * kD;
        for (int i = tid; i < kN * (kD / 8); i += kThreads) {
            const int h = i / (kD / 8), c = (i % (kD / 8)) * 8;
            const uint4 v = h < G ? *reinterpret_cast<const uint4 *>(qg + h * kD + c) : make_uint4(0, 0, 0, 0);
            *reinterpret_cast<uint4 *>(sm + kOffQ + (c >> 6) * (kN * 128) + sw128(h, c & 63)) = v;
        }
    }
    fence_async_smem();
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
    const uint32_t tmem = *tmem_slot;
    const uint32_t tS = tmem, tO = tmem + kOcol;

    if (warp == 4) {
        // ---------------- TMA producer
        if (lane == 0) {
            while (ld_p < np) {
                const int st = ld_J % kNst;  // ld_J >= kNst here: the first kNst loads went out above
                if (!mbar_wait(empty(st), ((ld_J / kNst) - 1) & 1, abort_flag)) break;
                issue_next();
            }
            // drain: the last phase issued on each stage must have landed before the CTA exits,
            // also after an abort (mbar_drain does not give up when the abort flag is set)
            for (int j = ld_J - 1; j >= 0 && j >= ld_J - kNst; --j) mbar_drain(full(j % kNst), (j / kNst) & 1);
        }
        __syncwarp();
    } else if (warp == 5) {
        // ---------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t id_qk = idesc_bf16(false, 128, kN);
            constexpr uint32_t id_pv = idesc_bf16(true, 128, kN);
            // the new token's K (which = 0) or V (1) row over tile row r of ring stage st, in
            // the 128-byte swizzle the TMA wrote; the proxy fence orders the stores before the
            // MMAs that read the stage
            auto patch_new_row = [&](int st, int r, int which) {
                const uint4 *src = reinterpret_cast<const uint4 *>(sm + kOffNew) + which * 16;
                unsigned char *tile = sm + st * kStage;
#pragma unroll
                for (int c = 0; c < 16; ++c)
                    *reinterpret_cast<uint4 *>(tile + (c >> 3) * kHalf + r * 128 + ((((c & 7) ^ r) & 7) << 4)) = src[c];
                fence_async_smem();
            };
            bool ok = true;
            int J = 0, Q = 0;  // loads and P tiles consumed so far
            if (a.stall) ok = mbar_wait(stall_bar, 0, abort_flag, kStallNs);  // runs out: abort
            for (int p = 0; p < np && ok; ++p) {
                const int n = chunk_n(p);
                // the S tiles of the previous pass must have been read
                if (p > 0 && !(ok = mbar_wait(s_free, (p - 1) & 1, abort_flag))) break;
                fence_after_sync();
                for (int i = 0; i < n; ++i) {
                    const int st = (J + i) % kNst;
                    if (!(ok = mbar_wait(full(st), ((J + i) / kNst) & 1, abort_flag))) break;
                    fence_after_sync();
                    const int rn = p_new - (chunk_t0(p) + i * kTile);
                    if (p_new >= 0 && rn >= 0 && rn < kTile) patch_new_row(st, rn, 0);
                    const uint32_t ka = base + st * kStage;
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint64_t da = sdesc(ka + (kk >> 2) * kHalf + (kk & 3) * 32, 16, 1024);
                        const uint64_t db = sdesc(sQ + (kk >> 2) * (kN * 128) + (kk & 3) * 32, 16, 1024);
                        mma_bf16(tS + kN * i, da, db, id_qk, kk > 0 ? 1u : 0u);
                    }
                    mma_commit(empty(st));
                }
                if (!ok) break;
                J += n;
                mma_commit(s_full);
                // O of the previous pass must have been read before this pass overwrites it
                if (p > 0 && !(ok = mbar_wait(o_free, (p - 1) & 1, abort_flag))) break;
                for (int i = 0; i < n; ++i) {
                    const int st = (J + i) % kNst, q = Q + i;
                    if (!(ok = mbar_wait(full(st), ((J + i) / kNst) & 1, abort_flag))) break;
                    if (!(ok = mbar_wait(p_full(q & 1), (q >> 1) & 1, abort_flag))) break;
                    fence_after_sync();
                    const int rn = p_new - (chunk_t0(p) + i * kTile);
                    if (p_new >= 0 && rn >= 0 && rn < kTile) patch_new_row(st, rn, 1);
                    const uint32_t va = base + st * kStage;
                    const uint32_t pb = sP + (q & 1) * kOpBytes;
#pragma unroll
                    for (int kk = 0; kk < kTile / 16; ++kk) {
                        // A = V^T (MN-major): 64-dim atoms 16 KB apart (LBO), 8-token groups 1 KB apart (SBO)
                        const uint64_t da = sdesc(va + kk * 2048, kHalf, 1024);
                        const uint64_t db = sdesc(pb + (kk >> 2) * (kN * 128) + (kk & 3) * 32, 16, 1024);
                        mma_bf16(tO, da, db, id_pv, (i > 0 || kk > 0) ? 1u : 0u);
                    }
                    mma_commit(empty(st));
                    mma_commit(p_empty(q & 1));
                }
                if (!ok) break;
                J += n;
                Q += n;
                mma_commit(o_full);
            }
            // also after an abort: no MMA may still write TMEM when it is freed
            mma_commit(mma_done);
            mbar_drain(mma_done, 0);
        }
        __syncwarp();
    } else {
        // ---------------- softmax / epilogue: thread tid owns TMEM lane tid
        const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
        // running (max, sum) per head over the CTA's passes, and output dim tid of each head
        float M[G], W[G], acc[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            M[h] = -INFINITY;
            W[h] = 0.f;
            acc[h] = 0.f;
        }
        const int32_t *prow =
            a.pos ? a.pos + ((int64_t)b * a.rows_per_seq + (a.rows_per_seq == 1 ? 0 : g)) * a.cap : nullptr;
        const int64_t lbase = (((int64_t)b * a.sc_layers + a.sc_layer0 + li) * H + (int64_t)g * G) * a.lstride;
        bool ok = true;
        int Q = 0;  // P tiles written so far
        // Every bar.sync below runs once per pass in every softmax warp, whatever ok says.
        for (int p = 0; p < np; ++p) {
            const int n = chunk_n(p), t0 = chunk_t0(p);
            const int lo = max(t0, S0), t1 = min(t0 + n * kTile, S0 + L);  // the chunk's valid rows
            float mx[G], sum[G];
#pragma unroll
            for (int h = 0; h < G; ++h) {
                mx[h] = -INFINITY;
                sum[h] = 0.f;
            }
            // bit i: this thread's row of tile i is a valid, live slot.  The liveness of every
            // tile is fetched before the wait for the QK products, so its latency is hidden.
            uint32_t live_bits = 0u;
            for (int i = 0; i < n; ++i) {
                const int tok = t0 + i * kTile + tid;  // physical slot; logical slot tok - S0
                if (tok >= lo && tok < t1 && (!prow || __ldg(prow + (tok - S0)) >= 0)) live_bits |= 1u << i;
            }
            if (ok) ok = mbar_wait(s_full, p & 1, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            fence_after_sync();
            // sweep 1: chunk maximum (-inf for a head when every row of the chunk is dead)
            if (ok) {
                for (int i = 0; i < n; ++i) {
                    float v[NC];
                    tmem_ld<NC>(tS + lane_off + kN * i, v);
                    if ((live_bits >> i) & 1u) {
#pragma unroll
                        for (int h = 0; h < G; ++h) mx[h] = fmaxf(mx[h], v[h] * a.scale_log2);
                    }
                }
            }
            // chunk max per head over the 128 softmax threads
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float m = mx[h];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                if (lane == 0) red[warp * kN + h] = m;
            }
            __syncwarp();
            softmax_bar();
#pragma unroll
            for (int h = 0; h < G; ++h) mx[h] = fmaxf(fmaxf(red[h], red[kN + h]), fmaxf(red[2 * kN + h], red[3 * kN + h]));
            softmax_bar();

            // sweep 2: logits write-out, exp2, row sums and the P operand of each tile.  The
            // logits stores sit here, interleaved with the V stream; issued as a burst in
            // sweep 1 they measured slower.
            for (int i = 0; i < n && ok; ++i) {
                const int q = Q + i;
                if (q >= 2 && !(ok = __all_sync(0xffffffffu, mbar_wait(p_empty(q & 1), ((q >> 1) - 1) & 1, abort_flag))))
                    break;
                float v[NC];
                tmem_ld<NC>(tS + lane_off + kN * i, v);
                const int tok = t0 + i * kTile + tid;
                const bool valid = tok >= lo && tok < t1;
                const bool live = (live_bits >> i) & 1u;  // valid and not dead
                unsigned char *pbuf = sm + kOffP + (q & 1) * kOpBytes + (tid >> 6) * (kN * 128);
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float z = v[h] * a.scale_log2;
                    float pr = 0.f;
                    if (valid && a.logits && !a.gsum) a.logits[lbase + (int64_t)h * a.lstride + (tok - S0)] = live ? z : -INFINITY;
                    if (live) {  // mx[h] is finite here: it covers this row
                        pr = exp2f(z - mx[h]);
                        sum[h] += pr;
                    }
                    *reinterpret_cast<__nv_bfloat16 *>(pbuf + sw128(h, tid & 63)) = __float2bfloat16_rn(pr);
                }
                fence_async_smem();
                mbar_arrive(p_full(q & 1));
            }
            Q += n;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float t = sum[h];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
                if (lane == 0) red[warp * kN + h] = t;
            }
            __syncwarp();
            softmax_bar();
#pragma unroll
            for (int h = 0; h < G; ++h) sum[h] = red[h] + red[kN + h] + red[2 * kN + h] + red[3 * kN + h];
            if (p + 1 < np) softmax_bar();  // red is rewritten by the next pass

            // sweep 3 (single-chunk units): the chunk's max and sum are the unit's, so each row's
            // normalised probabilities are final; their sum over the KV head's query group is
            // stored per token.  The S tiles are still in TMEM (the PV products go to O).
            if (a.gsum && a.logits && ok) {
                if (ns_active == 1) {
                    float inv[G];
#pragma unroll
                    for (int h = 0; h < G; ++h) inv[h] = sum[h] > 0.f ? 1.f / sum[h] : 0.f;
                    const int64_t gbase = (((int64_t)b * a.sc_layers + a.sc_layer0 + li) * a.kv_heads + g) * a.lstride;
                    for (int i = 0; i < n; ++i) {
                        float v[NC];
                        tmem_ld<NC>(tS + lane_off + kN * i, v);
                        const int tok = t0 + i * kTile + tid;
                        if (tok >= lo && tok < t1) {
                            float gs = 0.f;
                            if ((live_bits >> i) & 1u) {
#pragma unroll
                                for (int h = 0; h < G; ++h) gs += exp2f(v[h] * a.scale_log2 - mx[h]) * inv[h];
                            }
                            a.logits[gbase + (tok - S0)] = gs;
                        }
                    }
                } else if (tid == 0) {
                    atomicOr(&g_tc_error, 2u);  // the host only asks for group sums when every unit has one chunk
                }
            }
            if (MP) {
                fence_before_sync();
                mbar_arrive(s_free);
            }

            if (ok) ok = mbar_wait(o_full, p & 1, abort_flag);
            ok = __all_sync(0xffffffffu, ok);
            fence_after_sync();
            float o[NC];
#pragma unroll
            for (int h = 0; h < NC; ++h) o[h] = 0.f;
            if (ok) tmem_ld<NC>(tO + lane_off, o);
            if (MP) {
                fence_before_sync();
                mbar_arrive(o_free);
                // fold the pass into the running (max, sum, output); a pass whose rows are
                // all dead (mx = -inf, sum = 0, O = 0) leaves them unchanged
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float mn = fmaxf(M[h], mx[h]);
                    if (mn != -INFINITY) {
                        const float a_old = exp2f(M[h] - mn), a_new = exp2f(mx[h] - mn);
                        acc[h] = acc[h] * a_old + o[h] * a_new;
                        W[h] = W[h] * a_old + sum[h] * a_new;
                        M[h] = mn;
                    }
                }
            } else {
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    M[h] = mx[h];
                    W[h] = sum[h];
                    acc[h] = o[h];
                }
            }
        }

        if (MP || nc_unit == 1) {
            // the unit's only CTA (always so in a multi-pass launch, whose CTAs take all of
            // their unit's chunks): its output and log-sum-exp need no merge
            if (ok) {
#pragma unroll
                for (int h = 0; h < G; ++h)
                    a.out[(((int64_t)li * a.batch + b) * H + (int64_t)g * G + h) * kD + tid] =
                        __float2bfloat16_rn(W[h] > 0.f ? acc[h] / W[h] : 0.f);
                if (tid < G) {
                    float mm = -INFINITY, ss = 0.f;
#pragma unroll
                    for (int h = 0; h < G; ++h)
                        if (h == tid) {
                            mm = M[h];
                            ss = W[h];
                        }
                    a.lse2[((int64_t)b * a.sc_layers + a.sc_layer0 + li) * H + (int64_t)g * G + tid] =
                        ss > 0.f ? mm + log2f(ss) : -INFINITY;
                }
            }
        } else {
            const int64_t pbase = (((int64_t)b * a.n_layers + li) * H + (int64_t)g * G) * a.n_splits;
            if (ok) {
#pragma unroll
                for (int h = 0; h < G; ++h) a.part_o[((pbase + (int64_t)h * a.n_splits) + cta) * kD + tid] = acc[h];
                if (tid < G) {
                    float mm = -INFINITY, ss = 0.f;
#pragma unroll
                    for (int h = 0; h < G; ++h)
                        if (h == tid) {
                            mm = M[h];
                            ss = W[h];
                        }
                    a.part_ml[((pbase + (int64_t)tid * a.n_splits) + cta) * 2 + 0] = mm;
                    a.part_ml[((pbase + (int64_t)tid * a.n_splits) + cta) * 2 + 1] = ss;
                }
            }
            // The last CTA of (sequence, layer, kv head) to finish merges every CTA's
            // partial into the output and the per-head log-sum-exp.  Arrival counter
            // only: no CTA waits for another.
            softmax_bar();
            int *last_flag = reinterpret_cast<int *>(sm + kOffMisc + 8);
            const int64_t unit = ((int64_t)b * a.n_layers + li) * a.kv_heads + g;
            if (tid == 0) *last_flag = arrive_acq_rel(a.arrivals + unit) == nc_unit - 1 ? 1 : 0;
            softmax_bar();
            if (*last_flag && ok) {
                // partial weights [G][n_splits] in the P buffers (every MMA has completed)
                float *wq = reinterpret_cast<float *>(sm + kOffP);
                // warp w merges heads w, w + 4: (1) the partials' (max, sum) pairs give the
                // head's maximum M, each partial's weight exp2(m - M) (0 for one whose rows are
                // all dead) and the total W; (2) lane i sums the weighted partial outputs of
                // dims 4i .. 4i+3.  All loads of a phase are independent, so the merge costs a
                // few L2 round trips whatever the number of partials.
                for (int h = warp; h < G; h += 4) {
                    const float2 *ml = reinterpret_cast<const float2 *>(a.part_ml) + pbase + (int64_t)h * a.n_splits;
                    // the first kEarlyChunks partial outputs are loaded together with the
                    // (max, sum) pairs: their addresses do not depend on the weights
                    const float4 *po =
                        reinterpret_cast<const float4 *>(a.part_o + (pbase + (int64_t)h * a.n_splits) * kD) + lane;
                    float4 ov0[kEarlyChunks];
#pragma unroll
                    for (int j = 0; j < kEarlyChunks; ++j)
                        ov0[j] = j < nc_unit ? __ldcg(po + (int64_t)j * (kD / 4)) : make_float4(0.f, 0.f, 0.f, 0.f);
                    float mv[kMaxSplits / 32], lv[kMaxSplits / 32];
                    float Mh = -INFINITY;
#pragma unroll
                    for (int k = 0; k < kMaxSplits / 32; ++k) {
                        const int q = lane + 32 * k;
                        const float2 x = q < nc_unit ? __ldcg(ml + q) : make_float2(-INFINITY, 0.f);
                        mv[k] = x.x;
                        lv[k] = x.y;
                        Mh = fmaxf(Mh, x.x);
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) Mh = fmaxf(Mh, __shfl_xor_sync(0xffffffffu, Mh, o));
                    const float mref = Mh == -INFINITY ? 0.f : Mh;
                    float Wh = 0.f;
#pragma unroll
                    for (int k = 0; k < kMaxSplits / 32; ++k) {
                        const int q = lane + 32 * k;
                        const float wk = exp2f(mv[k] - mref);
                        Wh += lv[k] * wk;
                        if (q < nc_unit) wq[h * a.n_splits + q] = wk;
                    }
#pragma unroll
                    for (int o = 16; o > 0; o >>= 1) Wh += __shfl_xor_sync(0xffffffffu, Wh, o);
                    __syncwarp();
                    float4 sacc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int j = 0; j < kEarlyChunks; ++j) {
                        const float wj = j < nc_unit ? wq[h * a.n_splits + j] : 0.f;
                        sacc.x += wj * ov0[j].x;
                        sacc.y += wj * ov0[j].y;
                        sacc.z += wj * ov0[j].z;
                        sacc.w += wj * ov0[j].w;
                    }
                    for (int q0 = kEarlyChunks; q0 < nc_unit; q0 += 8) {
                        float4 ov[8];
#pragma unroll
                        for (int j = 0; j < 8; ++j)
                            ov[j] = q0 + j < nc_unit ? __ldcg(po + (int64_t)(q0 + j) * (kD / 4))
                                                     : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                        for (int j = 0; j < 8; ++j) {
                            const float wj = q0 + j < nc_unit ? wq[h * a.n_splits + q0 + j] : 0.f;
                            sacc.x += wj * ov[j].x;
                            sacc.y += wj * ov[j].y;
                            sacc.z += wj * ov[j].z;
                            sacc.w += wj * ov[j].w;
                        }
                    }
                    const bool any = Wh > 0.f;  // false only if every slot of the unit is dead
                    __nv_bfloat162 r0 = __floats2bfloat162_rn(any ? sacc.x / Wh : 0.f, any ? sacc.y / Wh : 0.f);
                    __nv_bfloat162 r1 = __floats2bfloat162_rn(any ? sacc.z / Wh : 0.f, any ? sacc.w / Wh : 0.f);
                    uint2 packed;
                    packed.x = *reinterpret_cast<uint32_t *>(&r0);
                    packed.y = *reinterpret_cast<uint32_t *>(&r1);
                    *reinterpret_cast<uint2 *>(a.out + (((int64_t)li * a.batch + b) * H + (int64_t)g * G + h) * kD +
                                               4 * lane) = packed;
                    if (lane == 0)
                        a.lse2[((int64_t)b * a.sc_layers + a.sc_layer0 + li) * H + (int64_t)g * G + h] =
                            any ? Mh + log2f(Wh) : -INFINITY;
                }
                if (tid == 0) a.arrivals[unit] = 0;
            }
        }
    }
    fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        fence_after_sync();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        cudaDriverEntryPointQueryResult q;
        void *p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool make_map(CUtensorMap *m, const void *pool, uint64_t rows, int rows_per_box) {
    auto fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {(cuuint64_t)kD, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)kD * 2};
    cuuint32_t box[2] = {64u, (cuuint32_t)rows_per_box};
    cuuint32_t es[2] = {1u, 1u};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(pool), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int G, bool MP>
cudaError_t launch_tc_gm(const CUtensorMap &mk, const CUtensorMap &mv, const TcArgs &t, dim3 grid, cudaStream_t st) {
    static bool attr = false;
    if (!attr) {
        cudaError_t e = cudaFuncSetAttribute(attend_tc_kernel<G, MP>, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    return launch_k(attend_tc_kernel<G, MP>, grid, dim3(kThreads), kSmemBytes, st, mk, mv, t);
}
template <int G>
cudaError_t launch_tc_g(const CUtensorMap &mk, const CUtensorMap &mv, const TcArgs &t, dim3 grid, cudaStream_t st) {
    return t.passes > 1 ? launch_tc_gm<G, true>(mk, mv, t, grid, st) : launch_tc_gm<G, false>(mk, mv, t, grid, st);
}

}  // namespace

int tc_max_split_tokens() { return kMaxTiles * kTile; }

#ifndef IKV_TC_WAVES
#define IKV_TC_WAVES 1
#endif
// shortest chunk of a single-wave launch (one layer of a small batch); at 8 units x 27
// tiles the split step measured 368 / 356 / 372 / 440 us per 32-layer step for 1 / 2 / 3 /
// 5 tiles
#ifndef IKV_TC_MIN_TILES
#define IKV_TC_MIN_TILES 2
#endif
// Chunking of the flattened (unit, tile) work for lengths up to max_len: enough
// chunks for about IKV_TC_WAVES waves of two CTAs per SM, each chunk 1..15 tiles,
// at most kMaxSplits chunks per unit.  Measured at 32 layers x 8 KV heads x 27 tiles:
// one wave's worth (chunks capped at 15 tiles, 512 CTAs) 77.3 us, two waves (12 tiles,
// 768 CTAs) 81.2 us, three 83.2 us, four 87.1 us -- fewer, longer CTAs spend less on
// prologues and merges.
void tc_plan(int32_t max_len, int64_t units, int sms, int32_t *item_tiles, int32_t *n_chunks) {
    const int64_t tiles = ((int64_t)max_len + kTile - 1) / kTile;
    const int64_t target = (int64_t)2 * sms * IKV_TC_WAVES;
    int64_t c = (units * tiles + target - 1) / target;
    // A launch with few units (one layer of a small batch) whose chunks fit a single wave
    // of resident CTAs takes the shortest chunks that still fit it: every CTA runs from
    // the start and no short tail wave follows.
    const int64_t per_unit = (int64_t)2 * sms / (units > 0 ? units : 1);
    if (per_unit >= 1 && (tiles + per_unit - 1) / per_unit <= kMaxTiles) {
        c = (tiles + per_unit - 1) / per_unit;
        if (c < IKV_TC_MIN_TILES) c = IKV_TC_MIN_TILES;
    }
    const int64_t cmin = (tiles + kMaxSplits - 1) / kMaxSplits;
    if (c < cmin) c = cmin;
    if (c < 1) c = 1;
    if (c > kMaxTiles) c = kMaxTiles;
    *item_tiles = (int32_t)c;
    const int64_t n = (tiles + c - 1) / c;
    *n_chunks = (int32_t)(n < 1 ? 1 : n);
}

bool tc_supported(int dtype, int head_dim, int group, int page_size) {
    if (dtype != IKV_BF16 || head_dim != kD) return false;
    if (!(group == 1 || group == 2 || group == 4 || group == 7 || group == 8)) return false;
    if (page_size % 128 == 0) return true;
    return page_size >= 8 && 128 % page_size == 0;
}

#ifndef IKV_TC_PASSES
#define IKV_TC_PASSES 1
#endif
// Consecutive chunks per CTA.  When the launch's units nearly fill one wave of resident
// CTAs on their own but their chunks do not (each chunk is at most 15 tiles), one CTA per
// unit takes all of the unit's chunks as passes: no second wave and no cross-CTA merge.
int tc_passes(int64_t units, int n_chunks, int sms, bool gsum) {
    if (!IKV_TC_PASSES || gsum || n_chunks <= 1 || units <= 0) return 1;
    const int64_t slots = (int64_t)2 * sms;
    if (units > slots || units * 4 < slots * 3) return 1;
    return n_chunks;
}

std::atomic<int> g_stall_next{0};

cudaError_t launch_attend_tc(const AttendArgs &a, const TcOutputs &o, int group, int sms, cudaStream_t st) {
    const int rpb = a.pv.page_size >= kTile ? kTile : a.pv.page_size;
    // rows of every layer the launch can touch: [layers][num_pages][kv_heads][page_size]
    const uint64_t rows = (uint64_t)(a.layer0 + a.n_layers) * a.pv.num_pages * a.pv.kv_heads * a.pv.page_size;
    CUtensorMap mk, mv;
    if (!make_map(&mk, a.k, rows, rpb) || !make_map(&mv, a.v, rows, rpb)) return cudaErrorInvalidValue;
    TcArgs t{};
    t.len = a.len;
    t.block_table = a.pv.block_table;
    t.start = a.pv.start;
    t.num_pages = a.pv.num_pages;
    t.page_size = a.pv.page_size;
    t.max_pages = a.pv.max_pages;
    t.kv_heads = a.pv.kv_heads;
    t.rows_per_box = rpb;
    t.q = reinterpret_cast<const __nv_bfloat16 *>(a.q);
    t.batch = a.batch;
    t.q_heads = a.q_heads;
    t.layer0 = a.layer0;
    t.n_layers = a.n_layers;
    t.split_tokens = a.split_tokens;
    t.n_splits = a.n_splits;
    t.cap = a.cap;
    t.scale_log2 = a.scale_log2;
    t.logits = a.logits;
    t.lstride = a.lstride;
    t.part_ml = a.part_ml;
    t.part_o = a.part_o;
    t.out = reinterpret_cast<__nv_bfloat16 *>(o.out);
    t.lse2 = o.lse2;
    t.arrivals = o.arrivals;
    t.pos = a.pos;
    t.rows_per_seq = a.rows_per_seq;
    t.sc_layers = a.sc_layers;
    t.sc_layer0 = a.sc_layer0;
    t.k_new = reinterpret_cast<const __nv_bfloat16 *>(a.k_new);
    t.v_new = reinterpret_cast<const __nv_bfloat16 *>(a.v_new);
    t.slot = a.slot;
    t.k_pool = reinterpret_cast<__nv_bfloat16 *>(const_cast<void *>(a.k));
    t.v_pool = reinterpret_cast<__nv_bfloat16 *>(const_cast<void *>(a.v));
    t.vnorm = a.vnorm;
    t.gsum = a.gsum;
    t.early = a.early;
    t.stall = g_stall_next.exchange(0);
    const int64_t units = (int64_t)a.pv.kv_heads * a.batch * a.n_layers;
    t.passes = tc_passes(units, a.n_splits, sms, a.gsum != 0);
    dim3 grid((unsigned)(((a.n_splits + t.passes - 1) / t.passes) * units));
    cudaError_t e;
    switch (group) {
        case 1: e = launch_tc_g<1>(mk, mv, t, grid, st); break;
        case 2: e = launch_tc_g<2>(mk, mv, t, grid, st); break;
        case 4: e = launch_tc_g<4>(mk, mv, t, grid, st); break;
        case 7: e = launch_tc_g<7>(mk, mv, t, grid, st); break;
        case 8: e = launch_tc_g<8>(mk, mv, t, grid, st); break;
        default: return cudaErrorInvalidValue;
    }
    note_launch();
    return e;
}

}  // namespace ikv

extern "C" ikv_status ikv_test_stall_next_attention(void) {
    ikv::g_stall_next.store(1);
    return IKV_OK;
}

extern "C" ikv_status ikv_device_status(uint32_t *flags) {
    if (!flags) return ikv::report(IKV_ERR_ARG, "flags is NULL");
    unsigned int v = 0, z = 0;
    cudaError_t e = cudaMemcpyFromSymbol(&v, ikv::g_tc_error, sizeof(v));
    if (e == cudaSuccess) e = cudaMemcpyToSymbol(ikv::g_tc_error, &z, sizeof(z));
    unsigned int ap = 0, lw = 0, tr = 0;
    if (e == cudaSuccess) e = ikv::read_clear_append_error(&ap);
    if (e == cudaSuccess) e = ikv::read_clear_layer_error(&lw);
    if (e == cudaSuccess) e = ikv::read_clear_trace_error(&tr);
    if (e != cudaSuccess) return ikv::report(IKV_ERR_CUDA, "ikv_device_status: %s", cudaGetErrorString(e));
    *flags = v | (ap ? 4u : 0u) | lw | tr;
    return IKV_OK;
}
