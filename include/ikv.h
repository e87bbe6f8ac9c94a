/*
 * ikv.h -- C ABI of the InertiaKV decode-step eviction path on GB300 (sm_103a).
 *
 * InertiaKV (arxiv 2609.03515) keeps, per sequence, a running utility m over
 * the cached tokens.  Every decode step appends the new token, runs grouped-
 * query decode attention, and (on refresh steps) folds each eligible layer's
 * head-averaged last-query attention probabilities into m with an EMA, layer
 * after layer.  Whenever the cache exceeds its budget B the lowest-utility
 * tokens are evicted for good and the surviving K/V rows are compacted.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every function returns ikv_status; IKV_OK == 0.  On error nothing is
 *    launched and ikv_last_error() returns a message (thread-local).
 *  - Tensor pointers are DEVICE pointers owned by the caller and borrowed for
 *    the duration of the call.  The library allocates and frees nothing;
 *    scratch memory comes from the caller's workspace (ws, ws_bytes), sized
 *    by the matching *_workspace_size function.  The workspace needs no
 *    initialisation and carries nothing between calls (ikv_params.ws_zeroed lets
 *    a caller that keeps one workspace for its steps skip the per-step zeroing).
 *  - Work is enqueued asynchronously on the caller's stream; arguments are
 *    checked on the host before anything is launched.  Errors raised by a
 *    kernel after launch surface as IKV_ERR_CUDA on a later call.
 *  - dtype of K/V/q/out: IKV_F32 or IKV_BF16.  Utilities, scores and all
 *    accumulation are fp32.  head_dim must be 64 or 128 and
 *    q_heads / kv_heads (the GQA group size G) one of 1, 2, 4, 7, 8.
 *  - Alignment: K/V pools, q, out, k_new, v_new must be 16-byte aligned.
 *  - bf16 pools with head_dim 128 and page_size 8..128 dividing 128 (or a
 *    multiple of 128) take the tensor-core attention path, which reads whole
 *    128-slot tiles: slots at or past len[b] inside a sequence's last tile
 *    must hold finite values (any finite values; zero-initialised pools and
 *    evicted rows qualify), and every block_table entry must name a valid page.
 *
 * Paged K/V layout
 * ----------------
 *  k, v: [layers][num_pages][kv_heads][page_size][head_dim] (dtype).
 *  Sequence b owns a slot space of cap = max_pages * page_size slots; slot p of
 *  it lives in physical page block_table[b][p / page_size] at offset
 *  p % page_size.  The sequence's cache slot j (j = 0..len[b]-1) is slot
 *  start[b] + j of that space (start == NULL means 0 for every sequence);
 *  start[b] + len[b] <= cap always.  Every block_table entry must name a valid
 *  page.
 *
 * Utility rows
 * ------------
 *  Granularity IKV_GRAN_SEQ (default): one utility row per sequence (rows =
 *  batch), Eq. 1 averages all q_heads, and the kept set applies to every
 *  layer and KV head.  IKV_GRAN_KVHEAD: one row per (sequence, KV head)
 *  (rows = batch * kv_heads, row index b * kv_heads + g), the score averages
 *  that KV head's query group, and the kept set applies to that KV head in
 *  every layer.  ema, pos and keep arrays are [rows][cap].
 *  Per-layer eviction (ikv_params.evict_mode = IKV_EVICT_LAYER, IKV_GRAN_SEQ):
 *  every layer keeps its own token set, so pos is [batch][layers][cap] (row
 *  b * layers + l lists layer l's positions by slot) and the utility is one
 *  state per token position: ema is [batch][pos_cap], indexed by position.
 */
#ifndef IKV_H
#define IKV_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    IKV_OK = 0,
    IKV_ERR_ARG = 1,         /* null pointer, out-of-range scalar */
    IKV_ERR_SHAPE = 2,       /* inconsistent or unsupported sizes */
    IKV_ERR_ALIGN = 3,       /* pointer not 16-byte aligned */
    IKV_ERR_WORKSPACE = 4,   /* workspace missing or too small */
    IKV_ERR_UNSUPPORTED = 5, /* valid request this build does not implement */
    IKV_ERR_CUDA = 6         /* a CUDA runtime call failed (incl. earlier async errors) */
} ikv_status;

enum { IKV_F32 = 0, IKV_BF16 = 1 };
enum { IKV_GRAN_SEQ = 0, IKV_GRAN_KVHEAD = 1 };
enum { IKV_COMPACT_STABLE = 0, IKV_COMPACT_HOLEFILL = 1, IKV_COMPACT_STABLE_SHORT = 2 };
enum { IKV_INIT_ZERO = 0, IKV_INIT_MEAN = 1 };
/* Temporal aggregation of the per-layer scores (Sec. 3.1): Eq. 4 EMA (InertiaKV),
 * Eq. 3 cumulative sum (H2O-style), Eq. 2 single-step. */
enum { IKV_AGG_EMA = 0, IKV_AGG_CUMULATIVE = 1, IKV_AGG_SINGLE_STEP = 2 };
/* Per-step scorer (Appendix "Per-step scoring"): Eq. 1 head-pooled attention; VNorm
 * (each head's probabilities times the l2 norm of the value row over the mean norm of
 * its (layer, kv head)); entropy weighting (each layer's pooled score times the
 * normalized entropy H(s) / ln n of that score over the n live slots, 1 if n = 1). */
enum { IKV_SCORE_ATTENTION = 0, IKV_SCORE_VNORM = 1, IKV_SCORE_ENTROPY = 2 };
/* When tokens are evicted: once per step after the last layer, one kept set for every
 * layer (default); or by every layer right after its own update of the state, from the
 * tokens that layer holds (Appendix "Layer scoring" hooks; layers' sets then differ). */
enum { IKV_EVICT_STEP = 0, IKV_EVICT_LAYER = 1 };

typedef struct {
    int32_t batch, layers, q_heads, kv_heads, head_dim;
    int32_t dtype;        /* IKV_F32 | IKV_BF16 */
    int32_t granularity;  /* IKV_GRAN_SEQ | IKV_GRAN_KVHEAD */
} ikv_shape;

typedef struct {
    void *k, *v;                 /* paged pools, see above (device) */
    const int32_t *block_table;  /* [batch][max_pages] physical page ids (device) */
    int32_t num_pages;           /* physical pages per layer in the pools */
    int32_t page_size;           /* slots per page, >= 1 */
    int32_t max_pages;           /* logical pages per sequence; cap = max_pages * page_size */
    int32_t *len;                /* [batch] slots in use per sequence (device); with dead_slots
                                    set this counts dead slots too */
    int32_t *pos;                /* [rows][cap] original token position per slot (device);
                                    -1 marks a dead slot (see dead_slots) */
    int32_t *next_pos;           /* [batch] position given to the next appended token (device) */
    int32_t max_len;             /* HOST-side upper bound on every len[b]; sizes launch grids */
    int32_t *start;              /* [batch] slot of cache slot 0 (device), or NULL = 0; moved
                                    only by IKV_COMPACT_STABLE_SHORT */
    int32_t dead_slots;          /* nonzero: slots whose pos is < 0 are dead -- evicted but not yet
                                    compacted away (ikv_params.max_holes).  Attention, scores,
                                    selection and the mean-utility append then skip them.
                                    0: every slot below len is live (pos is not read for it). */
    float *vnorm;                /* [layers][batch][kv_heads][cap] l2 norm of each cached value row,
                                    by logical slot (device), or NULL.  Needed by the VNorm scorer;
                                    when set, ikv_append_token / ikv_step store the new row's norm and
                                    compaction moves the norms with their rows.  Fill it once for the
                                    prefill with ikv_value_norms. */
    int32_t pos_cap;             /* per-layer eviction: token positions the position-indexed state
                                    holds (ema is [batch][pos_cap]; every next_pos[b] must stay below
                                    it); sizes the step workspace.  0 otherwise. */
} ikv_cache;

/* Optional per-kernel CUDA events recorded on the call's stream by ikv_step
 * (caller-created with cudaEventCreate; NULL members are skipped):
 * begin (before the append), append_end, attend_end (after the attention
 * kernel), combine_end (after the split combine), score_end (after the score
 * + EMA kernels), select_end, end (after compaction). */
typedef struct {
    cudaEvent_t begin, append_end, attend_end, combine_end, score_end, select_end, end;
} ikv_timing;

/* Rank-trace diagnostics (Appendix "Mechanistic Diagnostics"), an optional output of a
 * step, per utility row r:
 *  - raw top-k R_t: on refresh steps, the budget[b] tokens with the highest single-step
 *    score (the last eligible layer's score, the utility Eq. 2 would leave; ties to the
 *    lower slot), taken over the step's cache before eviction;
 *  - EMA top-k E_t: the tokens live after the step (the kept set).
 * Sets are token positions, ascending.  On entry raw_top / ema_top hold the previous
 * traced step's sets and n_top[r] = {|R_prev|, |E_prev|} (0, 0 before the first); on exit
 * this step's (raw_top and n_top[r][0] unchanged on steps without a raw score).
 * counts[r] = {|R_t & R_prev|, |E_t & E_prev|, |R_t & E_t|, |R_t|, |E_t|}, the R entries -1
 * on steps without a raw score.  Churn, Jaccard and the raw-top evicted fraction follow
 * from them.  A set larger than 16384 tokens is not traced: bit 4 of the device error
 * word, counts -2. */
typedef struct {
    int32_t *raw_top, *ema_top;  /* [rows][cap] device */
    int32_t *n_top;              /* [rows][2] device */
    int32_t *counts;             /* [rows][5] device, written */
} ikv_trace;

typedef struct {
    float alpha;                    /* EMA coefficient of Eq. 4, in [0, 1] */
    int32_t refresh_period;         /* r of Eq. 6 (>= 1; 1 = full refresh) */
    int32_t score_free;             /* 1: score at step 1 only, then freeze (Sec. 3.2) */
    const int32_t *budget;          /* [batch] decode budget B per sequence (device) */
    const uint8_t *layer_eligible;  /* HOST [layers] 0/1, NULL = all layers eligible */
    int32_t compact_mode;           /* IKV_COMPACT_STABLE (order-preserving, suffix moves left) |
                                       IKV_COMPACT_STABLE_SHORT (order-preserving, shorter side moves;
                                       needs cache->start) | IKV_COMPACT_HOLEFILL (set only) */
    int32_t refresh_init;           /* utility of a token appended on a refresh step:
                                       IKV_INIT_ZERO (m_0 = 0 rule) | IKV_INIT_MEAN */
    const ikv_timing *timing;       /* nullable */
    int32_t max_holes;              /* deferred compaction: 0 = compact on every eviction.  > 0:
                                       an evicted slot is only marked dead (pos = -1) while the
                                       sequence's dead slots stay <= max_holes; the step that
                                       would exceed it compacts (compact_mode) and clears them.
                                       The kept set and its order are the same either way; the
                                       attention reads up to max_holes extra (masked) slots, and
                                       rows move once per ~max_holes evictions instead of every
                                       step.  Needs pos; len then counts dead slots, so the
                                       caller's max_len bound is max(budget) + max_holes. */
    int32_t agg_mode;               /* how each eligible layer's score updates the utility, in layer
                                       order: IKV_AGG_EMA m = alpha m + (1 - alpha) s (Eq. 4, the
                                       method; default) | IKV_AGG_CUMULATIVE m = m + s (Eq. 3) |
                                       IKV_AGG_SINGLE_STEP m = s (Eq. 2) */
    int32_t scorer;                 /* IKV_SCORE_ATTENTION (Eq. 1, default) | IKV_SCORE_VNORM (needs
                                       cache->vnorm) | IKV_SCORE_ENTROPY */
    int32_t evict_mode;             /* IKV_EVICT_STEP (default) | IKV_EVICT_LAYER: each layer, after
                                       folding its score into the position-indexed state, keeps the
                                       budget[b] highest-utility tokens it holds (by the state as of its
                                       own update) and compacts its own rows (compact_mode; the shorter-
                                       side mode moves suffixes left).  A live position a layer does not
                                       hold scores 0 there, so its state decays by alpha (Eq. 1, Eq. 4);
                                       the mean initialisation averages the positions some layer holds.
                                       No layer's eviction changes another's inputs within a step, so the
                                       library applies them all after the step's attention (in ikv_step_end
                                       for the split step).  Needs IKV_GRAN_SEQ, max_holes 0, IKV_AGG_EMA,
                                       IKV_SCORE_ATTENTION, cache->pos_cap > 0 and the layout described
                                       under "Utility rows". */
    const ikv_trace *trace;         /* nullable: rank-trace diagnostics of the step (IKV_EVICT_STEP,
                                       scorer other than IKV_SCORE_ENTROPY) */
    int32_t ws_zeroed;              /* nonzero: the caller asserts that the workspace's control words
                                       are zero -- the workspace was zero-filled before its first step
                                       and every step since ran to completion with ikv_device_status()
                                       0 -- so ikv_step / ikv_step_begin skip re-zeroing them (two
                                       memset launches).  Every step leaves them zero. */
} ikv_params;

/* Message for the last error on this thread ("" if none). */
const char *ikv_last_error(void);

/* Number of kernels this library has launched in this process. */
int64_t ikv_launch_count(void);

/* Device-side error word of the current device, then cleared (synchronises
 * the device).  0 = no error.  Bit 0: a bounded wait inside the tensor-core
 * attention kernel ran out (the kernel abandoned its work and returned);
 * bit 1: a split longer than the kernel's TMEM budget reached the device;
 * bit 2: an append found no free slot (start + len = cap) and was dropped;
 * bit 3: per-layer eviction, a sequence's next_pos reached cache->pos_cap (the token
 * was dropped); bit 4: a rank-trace set exceeded 16384 tokens (not traced). */
ikv_status ikv_device_status(uint32_t *flags);

/* Test of the bounded waits (no counterpart in the paper): the next tensor-core attention
 * launch of this process starts with a wait, limited to 10 us, on a barrier that nothing
 * arrives at.  The wait runs out, so every CTA of that launch takes the timeout path --
 * abort flag, bit 0 of the device error word, its in-flight copies drained, TMEM freed --
 * and its outputs are undefined; later launches run normally.  Nothing faults or hangs.
 * Host only; launches nothing. */
ikv_status ikv_test_stall_next_attention(void);

/* Which decode-attention kernel ikv_decode_attend_score and ikv_step launch for
 * this shape and cache (all layers, cache->max_len):
 * IKV_PATH_TENSOR_CORE -- TMA-staged K/V tiles, tcgen05 QK^T and PV with TMEM
 *   accumulators; bf16, head_dim 128, group size 1, 2, 4, 7 or 8, page_size a
 *   divisor of 128 (>= 8) or a multiple of 128;
 * IKV_PATH_CUDA_CORE -- split-K flash decoding on the CUDA cores plus a combine
 *   kernel; every other supported shape.
 * Host only; launches nothing.  *path receives the value. */
enum { IKV_PATH_CUDA_CORE = 0, IKV_PATH_TENSOR_CORE = 1 };
ikv_status ikv_attend_path(const ikv_shape *shape, const ikv_cache *cache, int32_t *path);

/* How one attention launch over n_layers layers of every sequence (shape->layers: the
 * launch ikv_step makes; 1: a layer call of the split step) at lengths up to
 * cache->max_len is partitioned on a GPU with sms SMs (0: the current device's).  Each
 * (sequence, layer, KV head) unit's slots are cut into *n_chunks chunks of *chunk_tokens
 * slots (the tensor-core kernel sizes them for about one wave of two CTAs per SM, at
 * most 15 tiles of 128 slots); a CTA takes *passes consecutive chunks of its unit in turn
 * (more than 1 when the units alone nearly fill that wave but their chunks do not);
 * *group_sums is 1 when every unit is one chunk, so the launch hands the score pass
 * per-KV-head sums of normalised probabilities instead of per-head logits (Eq. 1 needs
 * only those).  *path as ikv_attend_path.  Host only; launches nothing.  Any output
 * pointer may be NULL; fails with IKV_ERR_ARG if n_layers is outside [1, layers] or
 * sms < 0. */
ikv_status ikv_attend_plan(const ikv_shape *shape, const ikv_cache *cache, int32_t n_layers, int32_t sms,
                           int32_t *path, int32_t *chunk_tokens, int32_t *n_chunks, int32_t *passes,
                           int32_t *group_sums);

/* ---------------------------------------------------------------------------
 * ikv_decode_attend_score -- one layer of decode attention plus its score.
 *
 * Eq. 1 and Appendix "Per-step scoring" (last query's attention weights,
 * mean-pooled over heads; GQA heads share their KV head).  For every sequence
 * b and query head h of layer `layer`:
 *     out[b][h] = softmax(q[b][h] . K_g^T / sqrt(d)) V_g  over slots 0..len[b]-1
 * with g = h / G.  If score != NULL it also writes, for i < len[b],
 *     score[r][i] = mean over the row's heads of softmax probability of slot i
 * (all q_heads for IKV_GRAN_SEQ, the KV head's group for IKV_GRAN_KVHEAD).
 * If ema != NULL the EMA of Eq. 4 is applied in place for i < len[b]:
 *     ema[r][i] = alpha * ema[r][i] + (1 - alpha) * score_i
 * which is one layer of the Appendix's layer-sequential update.  With
 * cache->dead_slots set, dead slots (pos[r][i] < 0, r the row of (b, g)) are
 * left out of the softmax: their probability and score are 0.
 *
 *  q, out: [batch][q_heads][head_dim] (dtype).  score, ema: [rows][cap] fp32.
 *  ws: at least ikv_attend_workspace_size() bytes.
 * ------------------------------------------------------------------------- */
ikv_status ikv_attend_workspace_size(const ikv_shape *shape, const ikv_cache *cache, size_t *bytes);
ikv_status ikv_decode_attend_score(const ikv_shape *shape, const ikv_cache *cache, int32_t layer,
                                   const void *q, void *out, float *score, float *ema, float alpha,
                                   void *ws, size_t ws_bytes, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_decode_attend_score_static -- ikv_decode_attend_score without a
 * caller workspace.  The paper has no counterpart: this is for callers that
 * cannot allocate device memory (a runtime that hands out all device memory
 * up front and forbids later cudaMalloc, an operator hook inside a framework
 * that owns the allocator, a loop that cannot afford cudaMalloc's implicit
 * synchronisation).  It allocates nothing; its scratch is a fixed device
 * array inside the library of ikv_static_scratch_bytes() bytes (16 MiB),
 * held by every GPU that loads the library until the process exits.
 *  - Arguments and results are those of ikv_decode_attend_score.
 *  - Shapes whose scratch (ikv_attend_workspace_size) exceeds the array are
 *    rejected with IKV_ERR_WORKSPACE and a message; nothing is launched.
 *  - The first call on a device looks up the array's device address (with
 *    that device current) and keeps it for the life of the process; make that
 *    first call before any stream capture.  After cudaDeviceReset the kept
 *    address is stale: do not call this entry point again in that process.
 *  - All calls share the one array, which keeps the last call's contents
 *    (nothing in it needs clearing).  Calls whose GPU work overlaps -- other
 *    streams or other host threads on the same device -- race on it; the
 *    caller must serialise them.
 * ------------------------------------------------------------------------- */
size_t ikv_static_scratch_bytes(void);
ikv_status ikv_decode_attend_score_static(const ikv_shape *shape, const ikv_cache *cache, int32_t layer,
                                          const void *q, void *out, float *score, float *ema, float alpha,
                                          cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_value_norms -- l2 norm of every cached value row (Appendix "Per-step
 * scoring", VNorm): cache->vnorm[l][b][g][j] = ||V[l][b][g][slot j]||_2 for every
 * layer l, sequence b, KV head g and logical slot j < len[b] (through start and the
 * block table).  Call once after the prefill; the append and compaction keep it
 * current from then on.  Fails with IKV_ERR_ARG if cache->vnorm is NULL.
 * ------------------------------------------------------------------------- */
ikv_status ikv_value_norms(const ikv_shape *shape, const ikv_cache *cache, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_ema_update -- Eq. 4 on a score array, in place.
 *     ema[r][i] = alpha * ema[r][i] + (1 - alpha) * score[r][i],  i < len[r / rows_per_seq]
 *  rows_per_seq: 1 for IKV_GRAN_SEQ, kv_heads for IKV_GRAN_KVHEAD.
 * ------------------------------------------------------------------------- */
ikv_status ikv_ema_update(int32_t rows, int32_t cap, float *ema, const float *score, const int32_t *len,
                          int32_t rows_per_seq, float alpha, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_select_budget -- which tokens survive (Sec. 3: evict the lowest m_t(i)
 * whenever the cache exceeds B).
 *
 * For row r with L = len[r / rows_per_seq] and B = budget[r / rows_per_seq],
 * the live slots are i < L (with pos != NULL: those with pos[r][i] >= 0; dead
 * slots are never kept).  If at most B slots are live, all of them are kept;
 * otherwise the B live slots with the largest util[r][i].  keep[r][0..n) lists
 * them in ascending slot order, keep_len[r] = n.  Ties keep the lower slot;
 * -0.0 equals +0.0; NaN ranks below every number.  Bit-exact: the result
 * depends only on the fp32 values.
 *  util: [rows][cap] fp32; pos: [rows][cap] int32 or NULL; keep: [rows][cap]
 *  int32; keep_len: [rows] int32.
 * ------------------------------------------------------------------------- */
ikv_status ikv_select_budget(int32_t rows, int32_t cap, const float *util, const int32_t *len,
                             int32_t rows_per_seq, const int32_t *budget, const int32_t *pos, int32_t *keep,
                             int32_t *keep_len, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_compact_kv -- in-place gather compaction after eviction ("cache
 * remapping" of the Appendix "Hook-level profiling" paragraph).
 *
 * For every sequence b, layer and KV head g (utility row r of (b, g)):
 * slot j of the compacted row holds what slot keep[r][j] held, j < keep_len[r].
 * The same gather is applied to pos and, if ema != NULL, to ema.  Afterwards
 * len[b] = keep_len[r].  IKV_COMPACT_STABLE preserves the survivors' order
 * (moves only the shifted suffix); IKV_COMPACT_HOLEFILL moves survivors that
 * sit at slots >= keep_len into the evicted slots below keep_len, keeping the
 * same set but not its order (fewer moved rows).  IKV_COMPACT_STABLE_SHORT
 * also preserves the order but moves whichever side of the evicted slots is
 * shorter: the suffix left (start unchanged) or the prefix right (start[b]
 * grows by the number evicted), chosen per sequence, and only while the slot
 * space keeps room for the next append (needs cache->start; sequences with
 * several utility rows always compact left).
 *  keep/keep_len as produced by ikv_select_budget.  ws: at least
 *  ikv_compact_workspace_size() bytes.
 * ------------------------------------------------------------------------- */
ikv_status ikv_compact_workspace_size(const ikv_shape *shape, const ikv_cache *cache, int32_t mode, size_t *bytes);
ikv_status ikv_compact_kv(const ikv_shape *shape, ikv_cache *cache, const int32_t *keep, const int32_t *keep_len,
                          float *ema, int32_t mode, void *ws, size_t ws_bytes, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_append_token -- add the new token of every sequence at slot len[b].
 *
 * Writes k_new/v_new ([layers][batch][kv_heads][head_dim]) into slot len[b]
 * of every layer, sets pos[r][len[b]] = next_pos[b], and gives the token the
 * utility 0 (init_mean == 0) or the mean utility of the existing live tokens
 * of its row (init_mean == 1, Appendix "New token insertion during non-refresh
 * steps"; dead slots excluded when cache->dead_slots).  Then len[b] += 1 and
 * next_pos[b] += 1.
 * Fails with IKV_ERR_SHAPE (host) if max_len + 1 > cap.
 * ------------------------------------------------------------------------- */
ikv_status ikv_append_token(const ikv_shape *shape, ikv_cache *cache, const void *k_new, const void *v_new,
                            float *ema, int32_t init_mean, void *ws, size_t ws_bytes, cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_step -- one whole decode step t (1-based) of InertiaKV / -Lazy /
 * Score-Free for every sequence of the batch:
 *   1. refresh = score_free ? (t == 1) : ((t - 1) % refresh_period == 0)   (Eq. 6)
 *   2. append the new token (utility: refresh_init on refresh steps, the mean
 *      of the existing utilities otherwise; Appendix "New token insertion")
 *   3. attention of every layer over all len[b] slots (the new token included)
 *   4. refresh steps only: for each eligible layer in ascending order,
 *      ema = alpha * ema + (1 - alpha) * s_layer  (Eq. 1, Eq. 4, Appendix
 *      "Layer scoring"; or Eq. 3 / Eq. 2 per agg_mode); off-refresh steps leave
 *      ema untouched (Eq. 6)
 *   5. if more than budget[b] slots are live: keep the budget[b] highest
 *      utilities and compact, or with max_holes > 0 mark the evicted slots dead
 *      until their number would exceed max_holes (Appendix "Eviction on
 *      non-refresh steps": also on off-refresh steps)
 *  q: [layers][batch][q_heads][head_dim]; k_new, v_new: [layers][batch][kv_heads][head_dim];
 *  out: [layers][batch][q_heads][head_dim] (all dtype).  ema: [rows][cap] fp32.
 *  cache->max_len bounds len[] BEFORE the append; the step needs max_len + 1 <= cap.
 *  After the step the caller should lower max_len to max(budget) (+ max_holes)
 *  if it tracks it.  With max_holes > 0 the step treats the cache as holding
 *  dead slots whatever cache->dead_slots says.
 * ------------------------------------------------------------------------- */
ikv_status ikv_step_workspace_size(const ikv_shape *shape, const ikv_cache *cache, size_t *bytes);
ikv_status ikv_step(const ikv_shape *shape, const ikv_params *params, ikv_cache *cache, float *ema, int32_t t,
                    const void *q, const void *k_new, const void *v_new, void *out, void *ws, size_t ws_bytes,
                    cudaStream_t stream);

/* ---------------------------------------------------------------------------
 * ikv_step_begin / ikv_step_layer / ikv_step_end -- ikv_step split at its layer
 * boundary, for a model that has layer l's q, k_new and v_new only after layer
 * l-1's attention output (Appendix "Layer scoring": the scores come from each
 * layer's attention inside the forward pass).  Calling
 *     ikv_step_begin(t); ikv_step_layer(t, 0); ...; ikv_step_layer(t, layers-1); ikv_step_end(t)
 * on one stream does what ikv_step(t) does with the same arguments (results equal
 * up to the rounding of the attention's split-K merge, which is partitioned per
 * layer here).  Between the calls the stream may run other work that leaves the
 * cache, ema and ws alone; the sequence may be captured in a CUDA graph.
 *  - ikv_step_begin: step 2's bookkeeping -- reserves slot len[b] for the new token
 *    (its position and utility, as ikv_append_token), len[b] += 1.  Its K/V rows
 *    are written by ikv_step_layer.
 *  - ikv_step_layer: writes k_new/v_new ([batch][kv_heads][head_dim], layer `layer`)
 *    into the reserved slot and runs that layer's attention (step 3; out, q:
 *    [batch][q_heads][head_dim]); on refresh steps an eligible layer also keeps its
 *    attention logits in ws.  Every layer is called once, in ascending order.
 *  - ikv_step_end: step 4 -- the kept scores of every eligible layer folded into ema
 *    in ascending layer order, which is the order Eq. 4 prescribes; nothing reads ema
 *    before the eviction -- and step 5 (selection, deferred or immediate compaction;
 *    under IKV_EVICT_LAYER every layer's own eviction).
 *  All three take the same shape, params, cache (max_len: the bound on len[]
 *  before the append, as for ikv_step), ema, t and ws (ikv_step_workspace_size
 *  bytes, which carries the step's state from call to call).  Argument errors are
 *  reported by the call that sees them; nothing is launched then, and the step
 *  cannot be continued.
 * ------------------------------------------------------------------------- */
ikv_status ikv_step_begin(const ikv_shape *shape, const ikv_params *params, ikv_cache *cache, float *ema, int32_t t,
                          void *ws, size_t ws_bytes, cudaStream_t stream);
ikv_status ikv_step_layer(const ikv_shape *shape, const ikv_params *params, ikv_cache *cache, float *ema, int32_t t,
                          int32_t layer, const void *q, const void *k_new, const void *v_new, void *out, void *ws,
                          size_t ws_bytes, cudaStream_t stream);
ikv_status ikv_step_end(const ikv_shape *shape, const ikv_params *params, ikv_cache *cache, float *ema, int32_t t,
                        void *ws, size_t ws_bytes, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* IKV_H */
