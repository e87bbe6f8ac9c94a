// Budgeted selection of one utility row by one CTA; used by the select kernel and by
// the score pass, whose last CTA of a row selects that row at once.  See select.cu.
#pragma once
#include "ikv_internal.cuh"

namespace ikv {
namespace {


constexpr int kSelThreads = 1024;

__device__ __forceinline__ uint32_t ord_key(float f) {
    uint32_t u = __float_as_uint(f);
    if ((u & 0x7FFFFFFFu) > 0x7F800000u) return 1u;  // NaN: below every number (-inf maps to 0x007FFFFF)
    if ((u & 0x7FFFFFFFu) == 0u) u = 0u;              // -0.0 == +0.0
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
constexpr uint32_t kDeadKey = 0u;  // dead slots: below every live key, never kept

// exclusive scan of one value per thread across a block of NT threads; returns (exclusive, total)
template <int NT>
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t *warp_tot, uint32_t &total) {
    constexpr int NW = NT / 32;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_tot[warp] = x;
    __syncthreads();
    if (warp == 0) {
        uint32_t t = lane < NW ? warp_tot[lane] : 0u;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(0xffffffffu, t, o);
            if (lane >= o) t += y;
        }
        if (lane < NW) warp_tot[lane] = t;  // inclusive over warps
    }
    __syncthreads();
    const uint32_t before = warp == 0 ? 0u : warp_tot[warp - 1];
    total = warp_tot[NW - 1];
    __syncthreads();
    return before + x - v;
}

// The selection of utility row r by the calling CTA, which must have NT threads (256 or
// 1024) and be entered by all of them.
template <int NT = kSelThreads>
__device__ __forceinline__ void select_row(int r, int32_t cap, const float *__restrict__ util,
                                           const int32_t *__restrict__ len, int32_t rps,
                                           const int32_t *__restrict__ budget, int32_t *pos, int32_t *keep,
                                           int32_t *keep_len, DeferArgs df) {
    static_assert(NT == 256 || NT == 1024, "the digit scan needs 256 threads at least, whole warps");
    constexpr int NW = NT / 32;
    __shared__ uint32_t hist[256];
    __shared__ uint32_t warp_tot[32];
    __shared__ unsigned long long s_min[32];
    __shared__ uint32_t s_digit, s_above, s_live;

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int L = len[r / rps];
    int B = budget[r / rps];
    if (B < 0) B = 0;
    const float *u = util + (int64_t)r * cap;
    int32_t *pr = pos ? pos + (int64_t)r * cap : nullptr;
    int32_t *kp = keep + (int64_t)r * cap;
    auto live = [&](int i) { return !pr || pr[i] >= 0; };
    auto key_at = [&](int i) { return live(i) ? ord_key(u[i]) : kDeadKey; };
    // every slot i < L for which keep_if(i) holds, in ascending order (block scans)
    auto write_kept = [&](auto keep_if) {
        uint32_t run = 0u;
        for (int base = 0; base < L; base += NT) {
            const int i = base + tid;
            const uint32_t kf = (i < L && keep_if(i)) ? 1u : 0u;
            uint32_t tot;
            const uint32_t at = block_excl_scan<NT>(kf, warp_tot, tot);
            if (kf) kp[run + at] = i;
            run += tot;
        }
    };

    // one pass: the live count and the lowest (key, highest slot) among the live slots,
    // which is the victim whenever exactly one slot must go
    if (tid == 0) s_live = 0u;
    __syncthreads();
    uint32_t c = 0u;
    unsigned long long best = ~0ull;
    for (int i = tid; i < L; i += NT) {
        if (!live(i)) continue;
        ++c;
        const unsigned long long v = ((unsigned long long)ord_key(u[i]) << 32) | (uint32_t)(~(uint32_t)i);
        best = v < best ? v : best;
    }
    if (pr && c) atomicAdd(&s_live, c);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
        best = y < best ? y : best;
    }
    if (lane == 0) s_min[warp] = best;
    __syncthreads();
    if (warp == 0) {
        best = lane < NW ? s_min[lane] : ~0ull;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const unsigned long long y = __shfl_xor_sync(0xffffffffu, best, o);
            best = y < best ? y : best;
        }
        if (lane == 0) s_min[0] = best;
    }
    __syncthreads();
    const int n_live = pr ? (int)s_live : L;

    if (n_live <= B) {
        if (n_live == L) {
            for (int j = tid; j < L; j += NT) kp[j] = j;
        } else {
            write_kept([&](int i) { return live(i); });
        }
        if (tid == 0) keep_len[r] = n_live;
        return;
    }
    if (B == 0) {
        if (tid == 0) keep_len[r] = 0;
        return;
    }

    if (n_live == B + 1) {
        const int ev = (int)(~(uint32_t)(s_min[0] & 0xFFFFFFFFull));
        const int b = r / rps;
        if (pr && df.max_holes > 0 && L - B <= df.max_holes && (df.start ? df.start[b] : 0) + L < df.cap) {
            // deferred compaction (the rule the compaction kernels apply): the victim is
            // only marked dead, and keep_len < 0 tells compaction that nothing moves
            if (tid == 0) {
                pr[ev] = -1;
                keep_len[r] = -1 - B;
            }
            return;
        }
        if (n_live == L) {
            for (int j = tid; j < B; j += NT) kp[j] = j < ev ? j : j + 1;
        } else {
            write_kept([&](int i) { return i != ev && live(i); });
        }
        if (tid == 0) keep_len[r] = B;
        return;
    }

    // general case: B < n_live - 1.  Dead slots carry the lowest key, and more than B
    // live keys lie above it, so the B-th largest key theta is live and no dead slot
    // is ever kept.
    uint32_t prefix = 0u, mask = 0u, k = (uint32_t)B;
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        for (int i = tid; i < 256; i += NT) hist[i] = 0u;
        __syncthreads();
        for (int base = 0; base < L; base += NT) {
            const int i = base + tid;
            uint32_t digit = 0xFFFFu;
            if (i < L) {
                const uint32_t key = key_at(i);
                if ((key & mask) == prefix) digit = (key >> shift) & 0xFFu;
            }
            const uint32_t peers = __match_any_sync(0xffffffffu, digit);
            if (digit != 0xFFFFu && lane == __ffs(peers) - 1) atomicAdd(&hist[digit], (uint32_t)__popc(peers));
        }
        __syncthreads();
        // inclusive counts from the top digit down: thread t < 256 holds digit 255 - t
        uint32_t v = 0u, x = 0u;
        if (tid < 256) {
            v = hist[255 - tid];
            x = v;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
                if (lane >= o) x += y;
            }
            if (lane == 31) warp_tot[warp] = x;
        }
        __syncthreads();
        if (tid < 256) {
            uint32_t before = 0u;
            for (int w = 0; w < warp; ++w) before += warp_tot[w];
            const uint32_t incl = before + x;
            const uint32_t above = incl - v;
            if (above < k && incl >= k) {  // exactly one digit satisfies this
                s_digit = 255u - (uint32_t)tid;
                s_above = above;
            }
        }
        __syncthreads();
        const uint32_t dsel = s_digit;
        k -= s_above;
        prefix |= dsel << shift;
        mask |= 0xFFu << shift;
        __syncthreads();
    }
    const uint32_t theta = prefix;
    const uint32_t need_eq = k;  // theta-valued slots that survive (lowest slots first)

    uint32_t run_eq = 0u, run_keep = 0u;
    for (int base = 0; base < L; base += NT) {
        const int i = base + tid;
        uint32_t key = 0u;
        bool in = i < L;
        if (in) key = key_at(i);
        const uint32_t gt = (in && key > theta) ? 1u : 0u;
        const uint32_t eq = (in && key == theta) ? 1u : 0u;
        uint32_t eq_tot, kp_tot;
        const uint32_t eq_rank = block_excl_scan<NT>(eq, warp_tot, eq_tot);
        const uint32_t kf = (gt || (eq && run_eq + eq_rank < need_eq)) ? 1u : 0u;
        const uint32_t at = block_excl_scan<NT>(kf, warp_tot, kp_tot);
        if (kf) kp[run_keep + at] = i;
        run_eq += eq_tot;
        run_keep += kp_tot;
    }
    if (tid == 0) keep_len[r] = B;
}

}  // namespace
}  // namespace ikv
