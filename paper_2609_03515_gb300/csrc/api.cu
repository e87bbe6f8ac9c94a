// C ABI of the InertiaKV decode-step path: argument checks, workspace layout
// and the launch sequence of one decode step.  No allocation happens here.
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <optional>

#include "ikv_internal.cuh"

namespace ikv {

static std::atomic<int64_t> g_launches{0};
static thread_local int g_pdl = 0;
bool pdl_enabled() { return g_pdl > 0; }
PdlScope::PdlScope() { ++g_pdl; }
PdlScope::~PdlScope() { --g_pdl; }
void note_launch(int n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

namespace {

thread_local char g_err[512] = "";

ikv_status fail(ikv_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

ikv_status cuda_fail(cudaError_t e, const char *what) {
    return fail(IKV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define IKV_TRY_CUDA(expr, what)                         \
    do {                                                 \
        cudaError_t _e = (expr);                         \
        if (_e != cudaSuccess) return cuda_fail(_e, what); \
    } while (0)

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int sm_count() {
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
        cached[dev] = n;
    }
    return cached[dev];
}

ikv_status check_shape(const ikv_shape *s) {
    if (!s) return fail(IKV_ERR_ARG, "shape is NULL");
    if (s->batch <= 0 || s->layers <= 0 || s->q_heads <= 0 || s->kv_heads <= 0)
        return fail(IKV_ERR_SHAPE, "batch/layers/heads must be positive");
    if (s->layers > kMaxLayers) return fail(IKV_ERR_SHAPE, "layers > %d", kMaxLayers);
    if (s->q_heads % s->kv_heads) return fail(IKV_ERR_SHAPE, "q_heads %% kv_heads != 0");
    const int G = s->q_heads / s->kv_heads;
    if (!(G == 1 || G == 2 || G == 4 || G == 7 || G == 8))
        return fail(IKV_ERR_UNSUPPORTED, "GQA group %d not supported (1, 2, 4, 7, 8)", G);
    if (s->head_dim != 64 && s->head_dim != 128) return fail(IKV_ERR_UNSUPPORTED, "head_dim must be 64 or 128");
    if (s->dtype != IKV_F32 && s->dtype != IKV_BF16) return fail(IKV_ERR_ARG, "dtype must be IKV_F32 or IKV_BF16");
    if (s->granularity != IKV_GRAN_SEQ && s->granularity != IKV_GRAN_KVHEAD)
        return fail(IKV_ERR_ARG, "granularity must be IKV_GRAN_SEQ or IKV_GRAN_KVHEAD");
    return IKV_OK;
}

int elem_bytes(const ikv_shape *s) { return s->dtype == IKV_BF16 ? 2 : 4; }
int rows_per_seq(const ikv_shape *s) { return s->granularity == IKV_GRAN_SEQ ? 1 : s->kv_heads; }

ikv_status check_cache(const ikv_shape *s, const ikv_cache *c, bool need_pos) {
    if (!c) return fail(IKV_ERR_ARG, "cache is NULL");
    if (!c->k || !c->v || !c->block_table || !c->len) return fail(IKV_ERR_ARG, "cache k/v/block_table/len is NULL");
    if (need_pos && (!c->pos || !c->next_pos)) return fail(IKV_ERR_ARG, "cache pos/next_pos is NULL");
    if (c->dead_slots && !c->pos) return fail(IKV_ERR_ARG, "dead_slots needs cache->pos");
    if (!aligned16(c->k) || !aligned16(c->v)) return fail(IKV_ERR_ALIGN, "K/V pools must be 16-byte aligned");
    if (c->page_size <= 0 || c->max_pages <= 0 || c->num_pages <= 0)
        return fail(IKV_ERR_SHAPE, "page_size/max_pages/num_pages must be positive");
    const int64_t cap = (int64_t)c->page_size * c->max_pages;
    if (cap > (int64_t)(1 << 30)) return fail(IKV_ERR_SHAPE, "cap too large");
    if (c->max_len < 0 || c->max_len > cap) return fail(IKV_ERR_SHAPE, "max_len %d outside [0, cap=%lld]", c->max_len, (long long)cap);
    (void)s;
    return IKV_OK;
}

int32_t cap_of(const ikv_cache *c) { return c->page_size * c->max_pages; }

PagedView view_of(const ikv_shape *s, const ikv_cache *c) {
    PagedView v;
    v.block_table = c->block_table;
    v.start = c->start;
    v.num_pages = c->num_pages;
    v.page_size = c->page_size;
    v.max_pages = c->max_pages;
    v.kv_heads = s->kv_heads;
    v.head_dim = s->head_dim;
    return v;
}

// ---- workspace layout ------------------------------------------------------
size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

int32_t logit_stride(int32_t cap) { return (cap + 127) / 128 * 128; }

struct AttendWs {
    size_t part_ml, part_o, lse2, arrivals, logits, end;
};

AttendWs attend_ws(const ikv_shape *s, int32_t cap, int n_layers, bool logits) {
    AttendWs w;
    size_t off = 0;
    const size_t bhl = (size_t)s->batch * n_layers * s->q_heads;
    w.part_ml = off;
    off = align256(off + bhl * kMaxSplits * 2 * sizeof(float));
    w.part_o = off;
    off = align256(off + bhl * kMaxSplits * s->head_dim * sizeof(float));
    w.lse2 = off;
    off = align256(off + bhl * sizeof(float));
    w.arrivals = off;
    off = align256(off + (size_t)s->batch * n_layers * s->kv_heads * sizeof(int32_t));
    w.logits = off;
    if (logits) off = align256(off + bhl * (size_t)logit_stride(cap) * sizeof(float));
    w.end = off;
    return w;
}

struct StepWs {
    AttendWs at;
    size_t keep, keep_len, done, cdone, sdone, moves, n_moves, sbuf, epart, vmean, slot, inv, util, live, raw, keep_raw,
        n_raw, raw_pos, sel_best, sel_cnt, end;
};

StepWs step_ws(const ikv_shape *s, int32_t cap, int32_t pos_cap) {
    StepWs w;
    w.at = attend_ws(s, cap, s->layers, true);
    size_t off = w.at.end;
    // utility rows; selection rows: one per utility row, or per (sequence, layer) under
    // per-layer eviction
    const size_t R = (size_t)s->batch * rows_per_seq(s);
    const size_t Rs = pos_cap > 0 && s->layers > rows_per_seq(s) ? (size_t)s->batch * s->layers : R;
    w.keep = off;
    off = align256(off + Rs * cap * sizeof(int32_t));
    w.keep_len = off;
    off = align256(off + Rs * sizeof(int32_t));
    // one control block: append arrivals [batch], compaction arrivals [batch], fused-
    // selection arrivals [rows]
    const size_t blk_max = ((size_t)cap + 31) / 32;
    w.done = off;
    w.cdone = off + (size_t)s->batch * sizeof(int32_t);
    w.sdone = off + 2 * (size_t)s->batch * sizeof(int32_t);
    off = align256(off + (2 * (size_t)s->batch + R) * sizeof(int32_t));
    w.moves = off;
    off = align256(off + Rs * cap * 2 * sizeof(int32_t));
    w.n_moves = off;
    off = align256(off + Rs * sizeof(int32_t));
    // scorer variants: entropy pass buffers and VNorm means
    w.sbuf = off;
    off = align256(off + R * s->layers * (size_t)logit_stride(cap) * sizeof(float));
    w.epart = off;
    off = align256(off + R * (s->layers + 1) * blk_max * sizeof(float));
    w.vmean = off;
    off = align256(off + (size_t)s->batch * s->layers * s->kv_heads * sizeof(float));
    w.slot = off;  // split step: each sequence's reserved slot
    off = align256(off + (size_t)s->batch * sizeof(int32_t));
    // per-layer eviction: every layer's position -> slot map, every layer's utilities by slot
    w.inv = off;
    if (pos_cap > 0) off = align256(off + (size_t)s->batch * s->layers * pos_cap * sizeof(int32_t));
    w.util = off;
    if (pos_cap > 0) off = align256(off + (size_t)s->batch * s->layers * cap * sizeof(float));
    w.live = off;
    if (pos_cap > 0) off = align256(off + (size_t)s->batch * ((pos_cap + 31) / 32) * sizeof(uint32_t));
    // rank trace: the single-step score, its top-k slots and their positions
    w.raw = off;
    off = align256(off + R * cap * sizeof(float));
    w.keep_raw = off;
    off = align256(off + R * cap * sizeof(int32_t));
    w.n_raw = off;
    off = align256(off + R * sizeof(int32_t));
    w.raw_pos = off;
    off = align256(off + R * cap * sizeof(int32_t));
    // fused selection: per score block, the lowest (key, slot) and the live count
    w.sel_best = off;
    off = align256(off + R * blk_max * sizeof(unsigned long long));
    w.sel_cnt = off;
    off = align256(off + R * blk_max * sizeof(uint32_t));
    w.end = off;
    return w;
}

template <typename T>
T *at(void *ws, size_t off) {
    return reinterpret_cast<T *>(reinterpret_cast<unsigned char *>(ws) + off);
}

// split-K partition for lengths up to max_len: enough CTAs to fill the GPU
// (ctas_per_sm x SMs), splits a multiple of `granule` tokens and at most
// `max_split` tokens long, at most kMaxSplits per (sequence, layer, kv head)
void choose_splits(const ikv_shape *s, int n_layers, int32_t max_len, int granule, int max_split,
                   int32_t *split_tokens, int32_t *n_splits, int sms) {
    const int64_t units = (int64_t)s->batch * n_layers * s->kv_heads;
    const int64_t want = (int64_t)sms * 4;
    int64_t splits = (want + units - 1) / units;
    const int64_t by_len = (max_len + kMinSplitTokens - 1) / kMinSplitTokens;
    if (splits > by_len) splits = by_len;
    const int64_t need = (max_len + max_split - 1) / max_split;
    if (splits < need) splits = need;
    if (splits > kMaxSplits) splits = kMaxSplits;
    if (splits < 1) splits = 1;
    int64_t st = (max_len + splits - 1) / splits;
    st = (st + granule - 1) / granule * granule;
    if (st < granule) st = granule;
    *split_tokens = (int32_t)st;
    int64_t ns = (max_len + st - 1) / st;
    if (ns < 1) ns = 1;
    *n_splits = (int32_t)ns;
}

// attention (+ combine) over layers [layer0, layer0 + n_layers)
// The tensor-core kernel serves bf16, d = 128, groups {1,2,4,7,8}, page sizes that tile
// 128 rows, and pools whose rows a 32-bit TMA coordinate reaches; the split-K CUDA-core
// kernel serves the rest.
static bool use_tc(const ikv_shape *s, const ikv_cache *c, int32_t layers_touched, int32_t max_len) {
    const int group = s->q_heads / s->kv_heads;
    const uint64_t pool_rows = (uint64_t)layers_touched * c->num_pages * s->kv_heads * c->page_size;
    return tc_supported(s->dtype, s->head_dim, group, c->page_size) &&
           (int64_t)max_len + 127 <= (int64_t)kMaxSplits * tc_max_split_tokens() && pool_rows < (1ull << 31);
}

// Whether an attention launch over n_layers layers at max_len writes normalised group sums
// (run_attend with a gsum request): the tensor-core kernel with one chunk per unit.
bool attend_gsum(const ikv_shape *s, const ikv_cache *c, int32_t n_layers, int32_t max_len) {
    if (!use_tc(s, c, s->layers, max_len)) return false;
    int32_t it = 0, nc = 0;
    tc_plan(max_len + 127, (int64_t)s->batch * n_layers * s->kv_heads, sm_count(), &it, &nc);
    return nc == 1;
}

ikv_status run_attend(const ikv_shape *s, const ikv_cache *c, int32_t layer0, int32_t n_layers, int32_t max_len,
                      const void *q, void *out, void *ws, const AttendWs &w, bool logits, int32_t *split_out,
                      int32_t *nsplit_out, cudaStream_t st, const ikv_timing *tm = nullptr,
                      bool counters_zeroed = false, int32_t sc_layers = 0, int32_t sc_layer0 = 0,
                      const AppendArgs *append = nullptr, bool *gsum = nullptr) {
    AttendArgs a{};
    a.k = c->k;
    a.v = c->v;
    a.pv = view_of(s, c);
    a.len = c->len;
    a.q = q;
    a.batch = s->batch;
    a.q_heads = s->q_heads;
    a.layer0 = layer0;
    a.n_layers = n_layers;
    const int group = s->q_heads / s->kv_heads;
    const bool tc = use_tc(s, c, layer0 + n_layers, max_len);
    if (tc) {
        int32_t it = 0, nc = 0;
        // a start offset may put the first valid row anywhere in its 128-slot tile
        tc_plan(max_len + 127, (int64_t)s->batch * n_layers * s->kv_heads, sm_count(), &it, &nc);
        a.split_tokens = it * 128;
        a.n_splits = nc;
        // one chunk per unit: the kernel can hand the score pass normalised group sums
        a.gsum = gsum && logits && nc == 1 && use_tc(s, c, s->layers, max_len) ? 1 : 0;
    } else
        choose_splits(s, n_layers, max_len, kTileTokens, 1 << 30, &a.split_tokens, &a.n_splits, sm_count());
    a.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)s->head_dim));
    a.logits = logits ? at<float>(ws, w.logits) : nullptr;
    if (gsum) *gsum = false;
    a.cap = cap_of(c);
    a.lstride = logit_stride(a.cap);
    a.part_ml = at<float>(ws, w.part_ml);
    a.part_o = at<float>(ws, w.part_o);
    a.pos = c->dead_slots ? c->pos : nullptr;
    a.rows_per_seq = rows_per_seq(s);
    a.sc_layers = sc_layers > 0 ? sc_layers : n_layers;
    a.sc_layer0 = sc_layer0;
    // split step: the new token's rows of this layer are stored by the tensor-core kernel
    // itself, or by a copy kernel ahead of the CUDA-core one
    if (append && tc) {
        a.k_new = append->k_new;
        a.v_new = append->v_new;
        a.slot = append->slot;
        a.vnorm = append->vnorm;
        // a later layer call reads nothing before its dependency wait that the kernels
        // still draining ahead of it (the previous layer calls, or the caller's work
        // between them) write: the step's bookkeeping ran in ikv_step_begin, and this
        // layer's cached rows change only through the launch itself
        a.early = layer0 > 0 ? 1 : 0;
    } else if (append) {
        IKV_TRY_CUDA(launch_append_rows(*append, st), "append rows launch");
    }
    if (tc) {
        // fused combine: the last split of each unit writes out and lse2
        int32_t *arr = at<int32_t>(ws, w.arrivals);
        if (!counters_zeroed)
            IKV_TRY_CUDA(cudaMemsetAsync(arr, 0, sizeof(int32_t) * (size_t)s->batch * n_layers * s->kv_heads, st),
                         "cudaMemsetAsync");
        TcOutputs o{out, at<float>(ws, w.lse2), arr};
        if (max_len > 0) IKV_TRY_CUDA(launch_attend_tc(a, o, group, sm_count(), st), "tensor-core attend launch");
        if (tm && tm->attend_end) IKV_TRY_CUDA(cudaEventRecord(tm->attend_end, st), "cudaEventRecord");
    } else {
        if (max_len > 0) IKV_TRY_CUDA(launch_attend(a, s->dtype, s->head_dim, group, st), "attend launch");
        if (tm && tm->attend_end) IKV_TRY_CUDA(cudaEventRecord(tm->attend_end, st), "cudaEventRecord");
        CombineArgs cb{};
        cb.len = c->len;
        cb.batch = s->batch;
        cb.q_heads = s->q_heads;
        cb.n_layers = n_layers;
        cb.split_tokens = a.split_tokens;
        cb.n_splits = a.n_splits;
        cb.head_dim = s->head_dim;
        cb.part_ml = a.part_ml;
        cb.part_o = a.part_o;
        cb.out = out;
        cb.lse2 = at<float>(ws, w.lse2);
        cb.sc_layers = a.sc_layers;
        cb.sc_layer0 = a.sc_layer0;
        IKV_TRY_CUDA(launch_combine(cb, s->dtype, st), "combine launch");
    }
    if (split_out) *split_out = a.split_tokens;
    if (nsplit_out) *nsplit_out = a.n_splits;
    if (gsum) *gsum = a.gsum != 0;
    return IKV_OK;
}

// Scorer-variant scratch of ikv_step (null for the per-layer entry points, which
// score with Eq. 1 only).
struct ScorerWs {
    float *sbuf = nullptr, *epart = nullptr, *vmean = nullptr;
};

// Selection run by the score pass's last CTA of each row (ikv_step, ikv_step_end).
struct SelectFuse {
    unsigned long long *best;  // [rows][blk_max]
    uint32_t *cnt;             // [rows][blk_max]
    int32_t *row_done;
    const int32_t *budget;
    int32_t *pos;
    int32_t *keep, *keep_len;
    DeferArgs df;
};

ikv_status run_score(const ikv_shape *s, const ikv_cache *c, int32_t n_layers, const int32_t *elig, int n_elig,
                     int32_t max_len, void *ws, const AttendWs &w, float alpha, float *ema, float *score,
                     cudaStream_t st, int32_t agg = IKV_AGG_EMA, int32_t scorer = IKV_SCORE_ATTENTION,
                     const ScorerWs &sw = ScorerWs{}, int32_t layer0 = 0, bool store_only = false,
                     const SelectFuse *fuse = nullptr, bool *fused = nullptr, bool gsum = false) {
    ScoreArgs base{};
    base.len = c->len;
    base.batch = s->batch;
    base.q_heads = s->q_heads;
    base.kv_heads = s->kv_heads;
    base.rows_per_seq = rows_per_seq(s);
    base.n_layers = n_layers;
    base.cap = cap_of(c);
    base.logits = at<float>(ws, w.logits);
    base.lstride = logit_stride(cap_of(c));
    base.lse2 = at<float>(ws, w.lse2);
    base.alpha = alpha;
    base.agg = agg;
    base.ema = ema;
    base.score = score;
    base.layer0 = layer0;
    base.scorer = scorer;
    base.vnorm = c->vnorm;
    base.vmean = sw.vmean;
    base.pos = c->dead_slots ? c->pos : nullptr;
    base.sbuf = sw.sbuf;
    base.epart = sw.epart;
    base.n_elig_total = n_elig;
    base.store_only = store_only ? 1 : 0;
    base.gsum = gsum ? 1 : 0;
    int V = 1;
    base.nblk = score_blocks(base, max_len, sm_count(), &V);
    base.blk_tok = 32 * V;
    if (scorer == IKV_SCORE_VNORM && !store_only) IKV_TRY_CUDA(launch_vnorm_mean(base, st), "vnorm mean launch");
    if (fused) *fused = false;
    for (int k0 = 0; k0 < n_elig; k0 += kMaxLayersPerScorePass) {
        ScoreArgs sa = base;
        sa.n_elig = n_elig - k0 < kMaxLayersPerScorePass ? n_elig - k0 : kMaxLayersPerScorePass;
        sa.k0 = k0;
        for (int k = 0; k < sa.n_elig; ++k) sa.elig[k] = elig[k0 + k];
        // the last pass of an Eq. 1 / VNorm fold also selects, unless the rows may be long
        // (step 1 after a long prefill): the general selection then runs in the 1024-thread
        // select kernel rather than on the score pass's last 256-thread CTA per row
        if (fuse && ema && !store_only && scorer != IKV_SCORE_ENTROPY && k0 + sa.n_elig == n_elig &&
            max_len <= kFusedSelectMaxLen) {
            sa.fuse_select = 1;
            sa.row_done = fuse->row_done;
            sa.budget = fuse->budget;
            sa.sel_pos = fuse->pos;
            sa.keep = fuse->keep;
            sa.keep_len = fuse->keep_len;
            sa.df = fuse->df;
            sa.sel_best = fuse->best;
            sa.sel_cnt = fuse->cnt;
            if (fused) *fused = true;
        }
        IKV_TRY_CUDA(launch_score_ema(sa, max_len, sm_count(), st), "score launch");
    }
    if (scorer == IKV_SCORE_ENTROPY && !store_only)
        IKV_TRY_CUDA(launch_entropy_fold(base, max_len, st), "entropy fold launch");
    return IKV_OK;
}

ikv_status record(cudaEvent_t e, cudaStream_t st) {
    if (e) IKV_TRY_CUDA(cudaEventRecord(e, st), "cudaEventRecord");
    return IKV_OK;
}

}  // namespace

ikv_status report(ikv_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return s;
}

}  // namespace ikv

using namespace ikv;

extern "C" {

const char *ikv_last_error(void) { return g_err; }

int64_t ikv_launch_count(void) { return g_launches.load(); }

ikv_status ikv_attend_workspace_size(const ikv_shape *shape, const ikv_cache *cache, size_t *bytes) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (!bytes) return fail(IKV_ERR_ARG, "bytes is NULL");
    *bytes = attend_ws(shape, cap_of(cache), 1, true).end;
    return IKV_OK;
}

ikv_status ikv_attend_path(const ikv_shape *shape, const ikv_cache *cache, int32_t *path) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (!path) return fail(IKV_ERR_ARG, "path is NULL");
    *path = use_tc(shape, cache, shape->layers, cache->max_len) ? IKV_PATH_TENSOR_CORE : IKV_PATH_CUDA_CORE;
    return IKV_OK;
}

ikv_status ikv_attend_plan(const ikv_shape *shape, const ikv_cache *cache, int32_t n_layers, int32_t sms,
                           int32_t *path, int32_t *chunk_tokens, int32_t *n_chunks, int32_t *passes,
                           int32_t *group_sums) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (n_layers < 1 || n_layers > shape->layers)
        return fail(IKV_ERR_ARG, "n_layers %d outside [1, %d]", n_layers, shape->layers);
    if (sms < 0) return fail(IKV_ERR_ARG, "sms must be >= 0");
    if (sms == 0) sms = sm_count();
    // the decisions run_attend and launch_attend_tc take for a launch from layer 0
    const int32_t max_len = cache->max_len;
    const int64_t units = (int64_t)shape->batch * n_layers * shape->kv_heads;
    const bool tc = use_tc(shape, cache, n_layers, max_len);
    int32_t ct = 0, nc = 0, np = 1, gs = 0;
    if (tc) {
        int32_t it = 0;
        tc_plan(max_len + 127, units, sms, &it, &nc);
        ct = it * 128;
        gs = nc == 1 && use_tc(shape, cache, shape->layers, max_len) ? 1 : 0;
        np = tc_passes(units, nc, sms, gs != 0);
    } else {
        choose_splits(shape, n_layers, max_len, kTileTokens, 1 << 30, &ct, &nc, sms);
    }
    if (path) *path = tc ? IKV_PATH_TENSOR_CORE : IKV_PATH_CUDA_CORE;
    if (chunk_tokens) *chunk_tokens = ct;
    if (n_chunks) *n_chunks = nc;
    if (passes) *passes = np;
    if (group_sums) *group_sums = gs;
    return IKV_OK;
}

ikv_status ikv_decode_attend_score(const ikv_shape *shape, const ikv_cache *cache, int32_t layer, const void *q,
                                   void *out, float *score, float *ema, float alpha, void *ws, size_t ws_bytes,
                                   cudaStream_t stream) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (layer < 0 || layer >= shape->layers) return fail(IKV_ERR_ARG, "layer %d out of range", layer);
    if (!q || !out) return fail(IKV_ERR_ARG, "q/out is NULL");
    if (!aligned16(q) || !aligned16(out)) return fail(IKV_ERR_ALIGN, "q/out must be 16-byte aligned");
    if (ema && !(alpha >= 0.f && alpha <= 1.f)) return fail(IKV_ERR_ARG, "alpha must be in [0, 1]");
    const bool want_score = score || ema;
    const AttendWs w = attend_ws(shape, cap_of(cache), 1, want_score);
    if (!ws || ws_bytes < w.end) return fail(IKV_ERR_WORKSPACE, "workspace needs %zu bytes", w.end);
    if ((e = run_attend(shape, cache, layer, 1, cache->max_len, q, out, ws, w, want_score, nullptr, nullptr, stream)))
        return e;
    if (want_score) {
        const int32_t elig0 = 0;
        if ((e = run_score(shape, cache, 1, &elig0, 1, cache->max_len, ws, w, ema ? alpha : 0.f, ema, score, stream)))
            return e;
    }
    return IKV_OK;
}

ikv_status ikv_value_norms(const ikv_shape *shape, const ikv_cache *cache, cudaStream_t stream) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (!cache->vnorm) return fail(IKV_ERR_ARG, "cache->vnorm is NULL");
    IKV_TRY_CUDA(launch_value_norms(cache->v, view_of(shape, cache), cache->len, shape->batch, shape->layers,
                                    cap_of(cache), shape->dtype, cache->vnorm, stream),
                 "value norms launch");
    return IKV_OK;
}

ikv_status ikv_ema_update(int32_t rows, int32_t cap, float *ema, const float *score, const int32_t *len,
                          int32_t rows_per_seq_, float alpha, cudaStream_t stream) {
    g_err[0] = 0;
    if (rows < 0 || cap < 0 || rows_per_seq_ <= 0) return fail(IKV_ERR_SHAPE, "rows/cap/rows_per_seq out of range");
    if (rows > 0 && (!ema || !score || !len)) return fail(IKV_ERR_ARG, "ema/score/len is NULL");
    if (!(alpha >= 0.f && alpha <= 1.f)) return fail(IKV_ERR_ARG, "alpha must be in [0, 1]");
    IKV_TRY_CUDA(launch_ema_update(rows, cap, ema, score, len, rows_per_seq_, alpha, cap, stream), "ema launch");
    return IKV_OK;
}

ikv_status ikv_select_budget(int32_t rows, int32_t cap, const float *util, const int32_t *len, int32_t rows_per_seq_,
                             const int32_t *budget, const int32_t *pos, int32_t *keep, int32_t *keep_len,
                             cudaStream_t stream) {
    g_err[0] = 0;
    if (rows < 0 || cap < 0 || rows_per_seq_ <= 0) return fail(IKV_ERR_SHAPE, "rows/cap/rows_per_seq out of range");
    if (rows > 0 && (!util || !len || !budget || !keep || !keep_len))
        return fail(IKV_ERR_ARG, "util/len/budget/keep/keep_len is NULL");
    // max_holes 0: the kernel never writes pos here
    IKV_TRY_CUDA(launch_select(rows, cap, util, len, rows_per_seq_, budget, const_cast<int32_t *>(pos), keep,
                               keep_len, DeferArgs{0, cap, nullptr}, stream),
                 "select launch");
    return IKV_OK;
}

ikv_status ikv_compact_workspace_size(const ikv_shape *shape, const ikv_cache *cache, int32_t mode, size_t *bytes) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (!bytes) return fail(IKV_ERR_ARG, "bytes is NULL");
    if (mode != IKV_COMPACT_STABLE && mode != IKV_COMPACT_HOLEFILL && mode != IKV_COMPACT_STABLE_SHORT)
        return fail(IKV_ERR_ARG, "unknown compact mode %d", mode);
    const size_t R = (size_t)shape->batch * rows_per_seq(shape);
    *bytes = align256((size_t)shape->batch * sizeof(int32_t));  // arrival counters
    if (mode == IKV_COMPACT_HOLEFILL)
        *bytes += align256(R * cap_of(cache) * 2 * sizeof(int32_t)) + align256(R * sizeof(int32_t));
    return IKV_OK;
}

static ikv_status compact_impl(const ikv_shape *shape, ikv_cache *cache, const int32_t *keep, const int32_t *keep_len,
                               float *ema, int32_t mode, int32_t *moves, int32_t *n_moves, int32_t *done,
                               cudaStream_t stream, int32_t max_holes = 0, bool by_layer = false) {
    CompactArgs a{};
    a.k = cache->k;
    a.v = cache->v;
    a.pv = view_of(shape, cache);
    a.batch = shape->batch;
    a.layers = shape->layers;
    a.rows_per_seq = rows_per_seq(shape);
    a.cap = cap_of(cache);
    a.elem_bytes = elem_bytes(shape);
    a.mode = mode;
    a.len = cache->len;
    a.pos = cache->pos;
    a.start = cache->start;
    a.done = done;
    a.ema = ema;
    a.keep = keep;
    a.keep_len = keep_len;
    a.moves = moves;
    a.n_moves = n_moves;
    a.max_holes = max_holes;
    a.vnorm = cache->vnorm;
    if (by_layer) {  // per-layer eviction: keep row (b, l) governs layer l's rows and pos row
        a.rows_per_seq = shape->layers;
        a.row_by_layer = 1;
    }
    IKV_TRY_CUDA(launch_compact(a, mode, sm_count(), stream), "compact launch");
    return IKV_OK;
}

ikv_status ikv_compact_kv(const ikv_shape *shape, ikv_cache *cache, const int32_t *keep, const int32_t *keep_len,
                          float *ema, int32_t mode, void *ws, size_t ws_bytes, cudaStream_t stream) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, true))) return e;
    if (!keep || !keep_len) return fail(IKV_ERR_ARG, "keep/keep_len is NULL");
    size_t need = 0;
    if ((e = ikv_compact_workspace_size(shape, cache, mode, &need))) return e;
    if (mode == IKV_COMPACT_STABLE_SHORT && !cache->start)
        return fail(IKV_ERR_ARG, "IKV_COMPACT_STABLE_SHORT needs cache->start");
    if (!ws || ws_bytes < need) return fail(IKV_ERR_WORKSPACE, "workspace needs %zu bytes", need);
    int32_t *done = at<int32_t>(ws, 0);
    const size_t off = align256((size_t)shape->batch * sizeof(int32_t));
    int32_t *moves = nullptr, *n_moves = nullptr;
    if (mode == IKV_COMPACT_HOLEFILL) {
        const size_t R = (size_t)shape->batch * rows_per_seq(shape);
        moves = at<int32_t>(ws, off);
        n_moves = at<int32_t>(ws, off + align256(R * cap_of(cache) * 2 * sizeof(int32_t)));
    }
    IKV_TRY_CUDA(cudaMemsetAsync(done, 0, sizeof(int32_t) * shape->batch, stream), "cudaMemsetAsync");
    return compact_impl(shape, cache, keep, keep_len, ema, mode, moves, n_moves, done, stream);
}

static ikv_status append_impl(const ikv_shape *shape, ikv_cache *cache, const void *k_new, const void *v_new,
                              float *ema, int32_t init_mean, int32_t *done, cudaStream_t stream,
                              bool counters_zeroed = false, int32_t *slot = nullptr) {
    AppendArgs a{};
    a.k = cache->k;
    a.v = cache->v;
    a.pv = view_of(shape, cache);
    a.batch = shape->batch;
    a.layers = shape->layers;
    a.rows_per_seq = rows_per_seq(shape);
    a.cap = cap_of(cache);
    a.elem_bytes = elem_bytes(shape);
    a.k_new = k_new;
    a.v_new = v_new;
    a.len = cache->len;
    a.pos = cache->pos;
    a.next_pos = cache->next_pos;
    a.ema = ema;
    a.init_mean = ema ? init_mean : 0;
    a.dead_slots = cache->dead_slots ? 1 : 0;
    a.done = done;
    a.vnorm = cache->vnorm;
    a.slot = slot;
    if (!counters_zeroed)
        IKV_TRY_CUDA(cudaMemsetAsync(done, 0, sizeof(int32_t) * shape->batch, stream), "cudaMemsetAsync");
    IKV_TRY_CUDA(launch_append(a, stream), "append launch");
    return IKV_OK;
}

ikv_status ikv_append_token(const ikv_shape *shape, ikv_cache *cache, const void *k_new, const void *v_new,
                            float *ema, int32_t init_mean, void *ws, size_t ws_bytes, cudaStream_t stream) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, true))) return e;
    if (!k_new || !v_new) return fail(IKV_ERR_ARG, "k_new/v_new is NULL");
    if (!aligned16(k_new) || !aligned16(v_new)) return fail(IKV_ERR_ALIGN, "k_new/v_new must be 16-byte aligned");
    if (cache->max_len + 1 > cap_of(cache)) return fail(IKV_ERR_SHAPE, "no free slot: max_len + 1 > cap");
    const size_t need = align256((size_t)shape->batch * sizeof(int32_t));
    if (!ws || ws_bytes < need) return fail(IKV_ERR_WORKSPACE, "workspace needs %zu bytes", need);
    return append_impl(shape, cache, k_new, v_new, ema, init_mean, at<int32_t>(ws, 0), stream);
}

// What every call of a decode step (ikv_step, or its begin / layer / end split) needs:
// checked arguments, the cache as the step's kernels see it, the workspace layout
// and the step's schedule.
struct StepCtx {
    ikv_cache cv;
    StepWs w;
    int32_t cap, L1, init_mean;
    bool scoring, layerwise;
    int32_t elig[kMaxLayers];
    int n_elig;
    ScorerWs sw;
};

static ikv_status prepare_step(const ikv_shape *shape, const ikv_params *p, const ikv_cache *cache, float *ema,
                               int32_t t, void *ws, size_t ws_bytes, StepCtx *cx) {
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, true))) return e;
    if (!p) return fail(IKV_ERR_ARG, "params is NULL");
    if (!ema || !p->budget) return fail(IKV_ERR_ARG, "ema/budget is NULL");
    if (t < 1) return fail(IKV_ERR_ARG, "t is 1-based (got %d)", t);
    if (!(p->alpha >= 0.f && p->alpha <= 1.f)) return fail(IKV_ERR_ARG, "alpha must be in [0, 1]");
    if (p->refresh_period < 1) return fail(IKV_ERR_ARG, "refresh_period must be >= 1");
    if (p->compact_mode != IKV_COMPACT_STABLE && p->compact_mode != IKV_COMPACT_HOLEFILL &&
        p->compact_mode != IKV_COMPACT_STABLE_SHORT)
        return fail(IKV_ERR_ARG, "unknown compact mode %d", p->compact_mode);
    if (p->compact_mode == IKV_COMPACT_STABLE_SHORT && !cache->start)
        return fail(IKV_ERR_ARG, "IKV_COMPACT_STABLE_SHORT needs cache->start");
    if (p->refresh_init != IKV_INIT_ZERO && p->refresh_init != IKV_INIT_MEAN)
        return fail(IKV_ERR_ARG, "unknown refresh_init %d", p->refresh_init);
    if (p->max_holes < 0) return fail(IKV_ERR_ARG, "max_holes must be >= 0");
    if (p->agg_mode != IKV_AGG_EMA && p->agg_mode != IKV_AGG_CUMULATIVE && p->agg_mode != IKV_AGG_SINGLE_STEP)
        return fail(IKV_ERR_ARG, "unknown agg_mode %d", p->agg_mode);
    if (p->scorer != IKV_SCORE_ATTENTION && p->scorer != IKV_SCORE_VNORM && p->scorer != IKV_SCORE_ENTROPY)
        return fail(IKV_ERR_ARG, "unknown scorer %d", p->scorer);
    if (p->scorer == IKV_SCORE_VNORM && !cache->vnorm) return fail(IKV_ERR_ARG, "IKV_SCORE_VNORM needs cache->vnorm");
    cx->layerwise = p->evict_mode == IKV_EVICT_LAYER;
    if (p->trace) {
        const ikv_trace *tr = p->trace;
        if (!tr->raw_top || !tr->ema_top || !tr->n_top || !tr->counts)
            return fail(IKV_ERR_ARG, "trace raw_top/ema_top/n_top/counts is NULL");
        if (cx->layerwise || p->scorer == IKV_SCORE_ENTROPY)
            return fail(IKV_ERR_UNSUPPORTED, "the rank trace needs IKV_EVICT_STEP and a scorer other than IKV_SCORE_ENTROPY");
    }
    if (p->evict_mode != IKV_EVICT_STEP && !cx->layerwise) return fail(IKV_ERR_ARG, "unknown evict_mode %d", p->evict_mode);
    if (cx->layerwise) {
        if (shape->granularity != IKV_GRAN_SEQ || p->max_holes != 0 || p->agg_mode != IKV_AGG_EMA ||
            p->scorer != IKV_SCORE_ATTENTION)
            return fail(IKV_ERR_UNSUPPORTED,
                        "IKV_EVICT_LAYER needs IKV_GRAN_SEQ, max_holes 0, IKV_AGG_EMA and IKV_SCORE_ATTENTION");
        if (cache->pos_cap <= 0) return fail(IKV_ERR_ARG, "IKV_EVICT_LAYER needs cache->pos_cap > 0");
        if (cache->dead_slots) return fail(IKV_ERR_ARG, "IKV_EVICT_LAYER does not use dead slots");
    }
    // with deferred compaction every kernel of the step treats pos < 0 as a dead slot
    cx->cv = *cache;
    if (p->max_holes > 0) cx->cv.dead_slots = 1;
    cx->cap = cap_of(cache);
    if (cache->max_len + 1 > cx->cap) return fail(IKV_ERR_SHAPE, "no free slot: max_len + 1 > cap");
    cx->w = step_ws(shape, cx->cap, cache->pos_cap);
    if (!ws || ws_bytes < cx->w.end) return fail(IKV_ERR_WORKSPACE, "workspace needs %zu bytes", cx->w.end);
    const bool refresh = p->score_free ? (t == 1) : ((t - 1) % p->refresh_period == 0);
    cx->n_elig = 0;
    for (int l = 0; l < shape->layers; ++l)
        if (!p->layer_eligible || p->layer_eligible[l]) cx->elig[cx->n_elig++] = l;
    cx->scoring = refresh && cx->n_elig > 0;
    cx->L1 = cache->max_len + 1;
    cx->init_mean = refresh ? (p->refresh_init == IKV_INIT_MEAN) : 1;
    cx->sw.sbuf = at<float>(ws, cx->w.sbuf);
    cx->sw.epart = at<float>(ws, cx->w.epart);
    cx->sw.vmean = at<float>(ws, cx->w.vmean);
    return IKV_OK;
}

// The step's counters -- attention arrivals, append / compaction / fused-selection
// arrivals -- zeroed, unless the caller vouches that they are (ikv_params.ws_zeroed).
static ikv_status zero_control_words(const ikv_params *p, void *ws, const StepWs &w, cudaStream_t stream) {
    if (p->ws_zeroed) return IKV_OK;
    IKV_TRY_CUDA(cudaMemsetAsync(at<int32_t>(ws, w.at.arrivals), 0, w.at.logits - w.at.arrivals, stream),
                 "cudaMemsetAsync");
    IKV_TRY_CUDA(cudaMemsetAsync(at<int32_t>(ws, w.done), 0, w.moves - w.done, stream), "cudaMemsetAsync");
    return IKV_OK;
}

// Step 5: selection, then deferred or immediate compaction.
static ikv_status evict_impl(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, void *ws,
                             const StepWs &w, cudaStream_t stream, const ikv_timing *tm, bool selected = false) {
    const int32_t cap = cap_of(cache);
    const int32_t R = shape->batch * rows_per_seq(shape);
    if (!selected)
        IKV_TRY_CUDA(launch_select(R, cap, ema, cache->len, rows_per_seq(shape), p->budget,
                                   cache->dead_slots ? cache->pos : nullptr, at<int32_t>(ws, w.keep),
                                   at<int32_t>(ws, w.keep_len), DeferArgs{p->max_holes, cap, cache->start}, stream),
                     "select launch");
    ikv_status e;
    if (tm && (e = record(tm->select_end, stream))) return e;
    return compact_impl(shape, cache, at<int32_t>(ws, w.keep), at<int32_t>(ws, w.keep_len), ema, p->compact_mode,
                        at<int32_t>(ws, w.moves), at<int32_t>(ws, w.n_moves), at<int32_t>(ws, w.cdone), stream,
                        p->max_holes);
}

// The selection the score pass may run itself (not under the rank trace, whose raw
// top-k must read the positions before the selection marks a victim dead).
static SelectFuse select_fuse(const ikv_params *p, const ikv_cache *cache, void *ws, const StepCtx &cx) {
    SelectFuse f;
    f.best = at<unsigned long long>(ws, cx.w.sel_best);
    f.cnt = at<uint32_t>(ws, cx.w.sel_cnt);
    f.row_done = at<int32_t>(ws, cx.w.sdone);
    f.budget = p->budget;
    f.pos = cache->dead_slots ? cache->pos : nullptr;
    f.keep = at<int32_t>(ws, cx.w.keep);
    f.keep_len = at<int32_t>(ws, cx.w.keep_len);
    f.df = DeferArgs{p->max_holes, cx.cap, cache->start};
    return f;
}

// Rank trace: the arguments of its kernels.
static TraceArgs trace_args(const ikv_shape *shape, const ikv_params *p, const ikv_cache *cache, void *ws,
                            const StepCtx &cx) {
    TraceArgs t{};
    t.rows = shape->batch * rows_per_seq(shape);
    t.rows_per_seq = rows_per_seq(shape);
    t.cap = cx.cap;
    t.len = cache->len;
    t.pos = cache->pos;
    t.keep_raw = at<int32_t>(ws, cx.w.keep_raw);
    t.n_raw = at<int32_t>(ws, cx.w.n_raw);
    t.raw_pos = at<int32_t>(ws, cx.w.raw_pos);
    t.has_raw = cx.scoring ? 1 : 0;
    t.raw_top = p->trace->raw_top;
    t.ema_top = p->trace->ema_top;
    t.n_top = p->trace->n_top;
    t.counts = p->trace->counts;
    return t;
}

// Rank trace, before the eviction: the raw top-k slots of the single-step score and
// their positions (refresh steps).
static ikv_status trace_before(const ikv_shape *shape, const ikv_params *p, const ikv_cache *cache, void *ws,
                               const StepCtx &cx, cudaStream_t stream) {
    if (!p->trace || !cx.scoring) return IKV_OK;
    const int32_t R = shape->batch * rows_per_seq(shape);
    IKV_TRY_CUDA(launch_select(R, cx.cap, at<float>(ws, cx.w.raw), cache->len, rows_per_seq(shape), p->budget,
                               cache->dead_slots ? cache->pos : nullptr, at<int32_t>(ws, cx.w.keep_raw),
                               at<int32_t>(ws, cx.w.n_raw), DeferArgs{0, cx.cap, nullptr}, stream),
                 "trace select launch");
    IKV_TRY_CUDA(launch_trace_gather(trace_args(shape, p, cache, ws, cx), cx.L1, stream), "trace gather launch");
    return IKV_OK;
}

static ikv_status trace_after(const ikv_shape *shape, const ikv_params *p, const ikv_cache *cache, void *ws,
                              const StepCtx &cx, cudaStream_t stream) {
    if (!p->trace) return IKV_OK;
    IKV_TRY_CUDA(launch_trace(trace_args(shape, p, cache, ws, cx), stream), "trace launch");
    return IKV_OK;
}

// Per-layer eviction: the arguments every layer-wise kernel of a step shares.
static LayerArgs layer_args(const ikv_shape *shape, const ikv_params *p, const ikv_cache *cache, float *ema, void *ws,
                            const StepCtx &cx) {
    LayerArgs a{};
    a.batch = shape->batch;
    a.layers = shape->layers;
    a.cap = cx.cap;
    a.pos_cap = cache->pos_cap;
    a.len = cache->len;
    a.next_pos = cache->next_pos;
    a.pos = cache->pos;
    a.start = cache->start;
    a.m = ema;
    a.inv = at<int32_t>(ws, cx.w.inv);
    a.util = at<float>(ws, cx.w.util);
    a.live = at<uint32_t>(ws, cx.w.live);
    a.live_words = (cache->pos_cap + 31) / 32;
    a.sbuf = cx.sw.sbuf;
    a.lstride = logit_stride(cx.cap);
    a.n_elig = cx.n_elig;
    a.alpha = p->alpha;
    a.scoring = cx.scoring ? 1 : 0;
    for (int k = 0; k < cx.n_elig; ++k) a.elig_bits[cx.elig[k] >> 5] |= 1u << (cx.elig[k] & 31);
    a.init_mean = cx.init_mean;
    a.slot = at<int32_t>(ws, cx.w.slot);
    return a;
}

// Per-layer eviction after every layer's attention: the eligible layers' pooled scores
// (refresh steps), the per-position fold giving each layer's utilities and the new
// state, then every (sequence, layer) row selected and every layer compacted at once.
static ikv_status layer_evict(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, void *ws,
                              const StepCtx &cx, cudaStream_t stream, bool gsum = false) {
    ikv_status e;
    if (cx.scoring && (e = run_score(shape, cache, shape->layers, cx.elig, cx.n_elig, cx.L1, ws, cx.w.at, p->alpha,
                                     nullptr, nullptr, stream, IKV_AGG_EMA, IKV_SCORE_ATTENTION, cx.sw, 0, true,
                                     nullptr, nullptr, gsum)))
        return e;
    IKV_TRY_CUDA(launch_layer_fold(layer_args(shape, p, cache, ema, ws, cx), cx.L1, cache->pos_cap, stream),
                 "layer fold launch");
    const int32_t K = shape->layers;
    IKV_TRY_CUDA(launch_select(shape->batch * K, cx.cap, at<float>(ws, cx.w.util), cache->len, K, p->budget, nullptr,
                               at<int32_t>(ws, cx.w.keep), at<int32_t>(ws, cx.w.keep_len), DeferArgs{0, cx.cap, nullptr},
                               stream),
                 "select launch");
    return compact_impl(shape, cache, at<int32_t>(ws, cx.w.keep), at<int32_t>(ws, cx.w.keep_len), nullptr,
                        p->compact_mode, at<int32_t>(ws, cx.w.moves), at<int32_t>(ws, cx.w.n_moves),
                        at<int32_t>(ws, cx.w.cdone), stream, 0, true);
}

ikv_status ikv_step_workspace_size(const ikv_shape *shape, const ikv_cache *cache, size_t *bytes) {
    g_err[0] = 0;
    ikv_status e = check_shape(shape);
    if (e) return e;
    if ((e = check_cache(shape, cache, false))) return e;
    if (!bytes) return fail(IKV_ERR_ARG, "bytes is NULL");
    *bytes = step_ws(shape, cap_of(cache), cache->pos_cap).end;
    return IKV_OK;
}

ikv_status ikv_step(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, int32_t t,
                    const void *q, const void *k_new, const void *v_new, void *out, void *ws, size_t ws_bytes,
                    cudaStream_t stream) {
    g_err[0] = 0;
    StepCtx cx;
    ikv_status e = prepare_step(shape, p, cache, ema, t, ws, ws_bytes, &cx);
    if (e) return e;
    if (!q || !k_new || !v_new || !out) return fail(IKV_ERR_ARG, "q/k_new/v_new/out is NULL");
    if (!aligned16(q) || !aligned16(out) || !aligned16(k_new) || !aligned16(v_new))
        return fail(IKV_ERR_ALIGN, "q/out/k_new/v_new must be 16-byte aligned");
    cache = &cx.cv;
    const StepWs &w = cx.w;
    const ikv_timing *tm = p->timing;
    if (cx.layerwise) {
        // begin, every layer's new rows, one attention launch for all layers (each reads
        // its own rows), then the per-layer evictions
        if ((e = zero_control_words(p, ws, w, stream))) return e;
        LayerArgs la = layer_args(shape, p, cache, ema, ws, cx);
        IKV_TRY_CUDA(cudaMemsetAsync(la.live, 0, sizeof(uint32_t) * (size_t)shape->batch * la.live_words, stream),
                     "cudaMemsetAsync");
        IKV_TRY_CUDA(launch_layer_begin(la, cache->max_len, stream), "layer begin launch");
        PdlScope pdl;
        AppendArgs ap{};
        ap.k = cache->k;
        ap.v = cache->v;
        ap.pv = view_of(shape, cache);
        ap.batch = shape->batch;
        ap.layers = shape->layers;
        ap.cap = cx.cap;
        ap.elem_bytes = elem_bytes(shape);
        ap.k_new = k_new;
        ap.v_new = v_new;
        ap.vnorm = cache->vnorm;
        ap.slot = at<int32_t>(ws, w.slot);
        IKV_TRY_CUDA(launch_append_rows(ap, stream), "append rows launch");
        bool gsum = false;
        if ((e = run_attend(shape, cache, 0, shape->layers, cx.L1, q, out, ws, w.at, cx.scoring, nullptr, nullptr,
                            stream, nullptr, true, 0, 0, nullptr, &gsum)))
            return e;
        return layer_evict(shape, p, cache, ema, ws, cx, stream, gsum);
    }

    // control words (append, split-arrival and selection counters) start at zero; every
    // kernel that counts leaves its counters zero again
    if ((e = zero_control_words(p, ws, w, stream))) return e;
    if (tm && (e = record(tm->begin, stream))) return e;
    // With the tensor-core attention the append is bookkeeping only (the new token's slot,
    // position and utility; len += 1, one CTA per sequence): the attention CTA whose chunk
    // holds the new slot stores that layer and KV head's rows itself and uses them in place
    // of the slot's old contents.  The CUDA-core path appends the rows first.
    const bool tc_rows = use_tc(shape, cache, shape->layers, cx.L1);
    int32_t *slot = at<int32_t>(ws, w.slot);
    if ((e = append_impl(shape, cache, tc_rows ? nullptr : k_new, tc_rows ? nullptr : v_new, ema, cx.init_mean,
                         at<int32_t>(ws, w.done), stream, true, tc_rows ? slot : nullptr)))
        return e;
    if (tm && (e = record(tm->append_end, stream))) return e;
    // the rest of the chain may overlap each kernel's ramp-up with its predecessor's tail
    // (not when per-kernel events are recorded: those time each kernel alone)
    std::optional<PdlScope> pdl;
    if (!tm) pdl.emplace();
    AppendArgs rows{};
    rows.k_new = k_new;
    rows.v_new = v_new;
    rows.slot = slot;
    rows.vnorm = cache->vnorm;
    bool gsum = false;  // the attention may hand over normalised group sums instead of logits
    if ((e = run_attend(shape, cache, 0, shape->layers, cx.L1, q, out, ws, w.at, cx.scoring, nullptr, nullptr, stream,
                        tm, true, 0, 0, tc_rows ? &rows : nullptr, &gsum)))
        return e;
    if (tm && (e = record(tm->combine_end, stream))) return e;
    float *raw = p->trace ? at<float>(ws, w.raw) : nullptr;
    const SelectFuse fs = select_fuse(p, cache, ws, cx);
    bool selected = false;
    if (cx.scoring && (e = run_score(shape, cache, shape->layers, cx.elig, cx.n_elig, cx.L1, ws, w.at, p->alpha, ema,
                                     raw, stream, p->agg_mode, p->scorer, cx.sw, 0, false,
                                     p->trace ? nullptr : &fs, &selected, gsum)))
        return e;
    if (tm && (e = record(tm->score_end, stream))) return e;
    if ((e = trace_before(shape, p, cache, ws, cx, stream))) return e;
    if ((e = evict_impl(shape, p, cache, ema, ws, w, stream, tm, selected))) return e;
    if (tm && (e = record(tm->end, stream))) return e;
    return trace_after(shape, p, cache, ws, cx, stream);
}

ikv_status ikv_step_begin(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, int32_t t,
                          void *ws, size_t ws_bytes, cudaStream_t stream) {
    g_err[0] = 0;
    StepCtx cx;
    ikv_status e = prepare_step(shape, p, cache, ema, t, ws, ws_bytes, &cx);
    if (e) return e;
    // control words start at zero (every kernel that counts leaves its counters zero)
    if ((e = zero_control_words(p, ws, cx.w, stream))) return e;
    if (cx.layerwise) {
        LayerArgs la = layer_args(shape, p, &cx.cv, ema, ws, cx);
        IKV_TRY_CUDA(cudaMemsetAsync(la.live, 0, sizeof(uint32_t) * (size_t)shape->batch * la.live_words, stream),
                     "cudaMemsetAsync");
        IKV_TRY_CUDA(launch_layer_begin(la, cache->max_len, stream), "layer begin launch");
        return IKV_OK;
    }
    return append_impl(shape, &cx.cv, nullptr, nullptr, ema, cx.init_mean, at<int32_t>(ws, cx.w.done), stream, true,
                       at<int32_t>(ws, cx.w.slot));
}

ikv_status ikv_step_layer(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, int32_t t,
                          int32_t layer, const void *q, const void *k_new, const void *v_new, void *out, void *ws,
                          size_t ws_bytes, cudaStream_t stream) {
    g_err[0] = 0;
    StepCtx cx;
    ikv_status e = prepare_step(shape, p, cache, ema, t, ws, ws_bytes, &cx);
    if (e) return e;
    if (layer < 0 || layer >= shape->layers) return fail(IKV_ERR_ARG, "layer %d out of range", layer);
    if (!q || !k_new || !v_new || !out) return fail(IKV_ERR_ARG, "q/k_new/v_new/out is NULL");
    if (!aligned16(q) || !aligned16(out) || !aligned16(k_new) || !aligned16(v_new))
        return fail(IKV_ERR_ALIGN, "q/out/k_new/v_new must be 16-byte aligned");
    cache = &cx.cv;
    PdlScope pdl;
    AppendArgs a{};
    a.k = cache->k;
    a.v = cache->v;
    a.pv = view_of(shape, cache);
    a.batch = shape->batch;
    a.layers = 1;
    a.rows_per_seq = rows_per_seq(shape);
    a.cap = cx.cap;
    a.elem_bytes = elem_bytes(shape);
    a.k_new = k_new;
    a.v_new = v_new;
    a.vnorm = cache->vnorm;
    a.layer0 = layer;
    a.slot = at<int32_t>(ws, cx.w.slot);
    bool eligible = false;
    for (int k = 0; k < cx.n_elig; ++k) eligible |= cx.elig[k] == layer;
    // the new token's rows and one layer's attention; on refresh steps its logits and
    // log-sum-exp land where the whole step's attention would put them, for
    // ikv_step_end's score pass
    bool gsum = false;  // the same for every layer call of the step (attend_gsum)
    return run_attend(shape, cache, layer, 1, cx.L1, q, out, ws, cx.w.at, cx.scoring && eligible, nullptr, nullptr,
                      stream, nullptr, true, shape->layers, layer, &a, &gsum);
}

ikv_status ikv_step_end(const ikv_shape *shape, const ikv_params *p, ikv_cache *cache, float *ema, int32_t t,
                        void *ws, size_t ws_bytes, cudaStream_t stream) {
    g_err[0] = 0;
    StepCtx cx;
    ikv_status e = prepare_step(shape, p, cache, ema, t, ws, ws_bytes, &cx);
    if (e) return e;
    PdlScope pdl;
    // what the layer calls' attention handed over: group sums when each launch had one chunk per unit
    const bool gsum = attend_gsum(shape, &cx.cv, 1, cx.L1);
    if (cx.layerwise) return layer_evict(shape, p, &cx.cv, ema, ws, cx, stream, gsum);
    float *raw = p->trace ? at<float>(ws, cx.w.raw) : nullptr;
    const SelectFuse fs = select_fuse(p, &cx.cv, ws, cx);
    bool selected = false;
    if (cx.scoring && (e = run_score(shape, &cx.cv, shape->layers, cx.elig, cx.n_elig, cx.L1, ws, cx.w.at, p->alpha,
                                     ema, raw, stream, p->agg_mode, p->scorer, cx.sw, 0, false,
                                     p->trace ? nullptr : &fs, &selected, gsum)))
        return e;
    if ((e = trace_before(shape, p, &cx.cv, ws, cx, stream))) return e;
    if ((e = evict_impl(shape, p, &cx.cv, ema, ws, cx.w, stream, nullptr, selected))) return e;
    return trace_after(shape, p, &cx.cv, ws, cx, stream);
}

}  // extern "C"
