// Internal declarations shared by the library's translation units.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "ikv.h"

namespace ikv {

constexpr int kTileTokens = 64;    // K/V rows staged per attention tile
constexpr int kAttendThreads = 128;
constexpr int kMaxSplits = 128;    // split-K partitions per (seq, layer, kv head)
constexpr int kMinSplitTokens = 256;
constexpr int kMaxLayersPerScorePass = 32;
constexpr int kFusedSelectMaxLen = 16384;  // longest row bound for which the score pass also selects
constexpr int kScoreLayersPerGroup = 8;   // eligible layers one score CTA folds (one warp each)
constexpr int kMaxLayers = 512;

// Launch-count bookkeeping (host).
void note_launch(int n = 1);

// Set the thread's ikv_last_error() message and return `s` (host).
ikv_status report(ikv_status s, const char *fmt, ...);

// Programmatic dependent launch.  While a PdlScope is alive on the issuing thread
// (ikv_step, for the kernels after its first), kernels are launched with programmatic
// stream serialisation: each may be scheduled while its predecessor drains.  Every
// kernel of the library starts with pdl_wait() -- which returns once all predecessor
// grids have completed and their memory is visible, and is a no-op for a normal launch
// -- before it reads or writes anything, then lets its own dependents be scheduled.
bool pdl_enabled();
struct PdlScope {
    PdlScope();
    ~PdlScope();
};
__device__ __forceinline__ void pdl_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
// A CTA's arrival on a counter shared by a group of CTAs, by one thread after a CTA
// barrier: an acquire-release add, so it releases the CTA's stores (the barrier orders
// the other threads' stores before it, and release is cumulative) and, for the last CTA
// to arrive, acquires every other CTA's before the barrier that follows.  Returns the
// count before the add.  (Measured: a gpu-scope fence on either side of a relaxed add
// cost ~0.4 us more per arrival chain.)
__device__ __forceinline__ int arrive_acq_rel(int *counter) {
    int before;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], 1;" : "=r"(before) : "l"(counter) : "memory");
    return before;
}
template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st, Args... args) {
    if (!pdl_enabled()) {
        kernel<<<grid, block, smem, st>>>(args...);
        return cudaGetLastError();
    }
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Where a (sequence, slot) row of layer l / kv head g lives in the paged pool.
// Logical slot j of sequence b is physical slot start[b] + j of its slot space
// [0, cap); physical slot p lives in page block_table[b][p / page_size].
struct PagedView {
    const int32_t *block_table;
    const int32_t *start;       // [batch] or null (all zero)
    int32_t num_pages, page_size, max_pages, kv_heads, head_dim;
    __device__ __forceinline__ int32_t start_of(int32_t b) const { return start ? start[b] : 0; }
    __device__ __forceinline__ int64_t row_phys(int32_t b, int32_t l, int32_t g, int32_t phys) const {
        const int32_t page = block_table[(int64_t)b * max_pages + phys / page_size];
        return (((int64_t)l * num_pages + page) * kv_heads + g) * page_size + phys % page_size;
    }
};

struct AttendArgs {
    const void *k, *v;          // pools
    PagedView pv;
    const int32_t *len;         // [batch]
    const void *q;              // q for layer layer0: element (li, b, h, e) at q + ((li*batch + b)*H + h)*D + e
    int32_t batch, q_heads, layer0, n_layers;
    int32_t split_tokens, n_splits;
    float scale_log2;           // log2(e) / sqrt(d)
    float *logits;              // [batch][sc_layers][H][lstride] log2-domain logits, or null
    int32_t cap;
    int32_t lstride;            // logits row stride: cap rounded up to a multiple of 128
    float *part_ml;             // [batch][n_layers][H][n_splits][2]  (running max, sum) in log2 domain
    float *part_o;              // [batch][n_layers][H][n_splits][D]  unnormalised partial output
    const int32_t *pos;         // [rows][cap] with -1 at dead slots, or null (every slot below len live)
    int32_t rows_per_seq;       // utility rows per sequence (row of (b, g): b * rows_per_seq + g or b)
    // logits and lse2 hold sc_layers layers per sequence; local layer li is their layer
    // sc_layer0 + li (a per-layer launch writes into a whole step's arrays)
    int32_t sc_layers, sc_layer0;
    // tensor-core kernel, split step: the new token's rows of this (single) layer,
    // [batch][kv_heads][D], stored into logical slot slot[b] (-1: none) before they are
    // read; their V norms into vnorm (or null).  k_new null: no append.
    const void *k_new, *v_new;
    const int32_t *slot;
    float *vnorm;
    // tensor-core kernel, every unit one chunk: logits holds, per token, each KV head's sum
    // of its query group's normalised probabilities ([batch][sc_layers][kv_heads][lstride])
    // instead of per-head logits
    int32_t gsum;
    // tensor-core kernel: the launch may set up and start its K/V stream before the
    // programmatic-dependency wait (see TcArgs::early)
    int32_t early;
};

struct CombineArgs {
    const int32_t *len;
    int32_t batch, q_heads, n_layers, split_tokens, n_splits, head_dim;
    const float *part_ml, *part_o;
    void *out;                  // [n_layers][batch][H][D] (dtype)
    float *lse2;                // [batch][sc_layers][H] log2-sum-exp, or null
    int32_t sc_layers, sc_layer0;
};

// Deferred compaction inside selection: when a row has exactly one slot too many and
// the sequence may defer (len - budget <= max_holes and start + len < cap), select
// marks the victim dead itself and writes keep_len = -1 - budget, which tells the
// compaction kernels that nothing moves.  max_holes = 0 disables it.
struct DeferArgs {
    int32_t max_holes;
    int32_t cap;
    const int32_t *start;       // [batch] or null
};

struct ScoreArgs {
    const int32_t *len;         // [batch]
    int32_t batch, q_heads, kv_heads, rows_per_seq, n_layers, cap;
    const float *logits;        // [batch][n_layers][H][lstride]
    int32_t lstride;
    const float *lse2;          // [batch][n_layers][H]
    int32_t n_elig;             // eligible local layers, in ascending order
    const int32_t *elig_dev;    // unused placeholder
    float alpha;
    int32_t agg;                // IKV_AGG_*: how each layer's score updates ema
    float *ema;                 // [rows][cap] or null
    float *score;               // [rows][cap] or null (only meaningful with one layer)
    int32_t elig[kMaxLayersPerScorePass];
    int32_t layer0;             // model layer of local layer 0 (vnorm indexing)
    int32_t scorer;             // IKV_SCORE_*
    const float *vnorm;         // VNorm: [layers][batch][kv_heads][cap] value-row norms
    float *vmean;               // VNorm: [batch][n_layers][kv_heads] mean norm over live slots
    const int32_t *pos;         // [rows][cap], -1 at dead slots, or null (all slots below len live)
    float *sbuf;                // entropy: [rows][n_elig_total][lstride] pooled scores
    float *epart;               // entropy: [rows][n_elig_total + 1][nblk] partial entropies, live counts
    int32_t nblk;               // entropy: token blocks of the score pass (partials row stride)
    int32_t blk_tok;            // entropy: tokens per block of the score pass
    int32_t k0;                 // eligible-layer index of this pass's first layer
    int32_t n_elig_total;       // eligible layers over all passes
    int32_t store_only;         // Eq. 1 scorer: only store each layer's pooled score in sbuf
    int32_t gsum;               // logits holds KV-head group sums of probabilities (see AttendArgs)
    // selection fused into the (last) pass: the last CTA of each row to finish its
    // utilities runs the budgeted selection of that row (select_row)
    int32_t fuse_select;
    int32_t *row_done;          // [rows] arrival counters, zero on entry, left zero
    const int32_t *budget;      // [batch]
    int32_t *sel_pos;           // pos when dead slots are in use, else null
    int32_t *keep, *keep_len;   // [rows][cap], [rows]
    DeferArgs df;
    unsigned long long *sel_best;  // [rows][nblk] each block's lowest (key, ~slot) among live slots
    uint32_t *sel_cnt;             // [rows][nblk] each block's live slots
};

// tensor-core attention (bf16, head_dim 128): attend_tc.cu
bool tc_supported(int dtype, int head_dim, int group, int page_size);
int tc_max_split_tokens();
// the tensor-core kernel also merges its splits (last CTA of each unit)
struct TcOutputs {
    void *out;                  // [n_layers][batch][H][128] bf16
    float *lse2;                // [batch][sc_layers][H]
    int32_t *arrivals;          // [batch][n_layers][kv_heads] zeroed before the launch
};
void tc_plan(int32_t max_len, int64_t units, int sms, int32_t *item_tiles, int32_t *n_chunks);
// consecutive chunks one CTA of the tensor-core kernel takes, for that chunk plan
int tc_passes(int64_t units, int n_chunks, int sms, bool gsum);
cudaError_t launch_attend_tc(const AttendArgs &a, const TcOutputs &o, int group, int sms, cudaStream_t st);

// launchers (return cudaError_t of the launch)
cudaError_t launch_attend(const AttendArgs &a, int dtype, int head_dim, int group, cudaStream_t st);
cudaError_t launch_combine(const CombineArgs &a, int dtype, cudaStream_t st);
cudaError_t launch_score_ema(const ScoreArgs &a, int32_t max_len, int sms, cudaStream_t st);
// token blocks (and tokens per lane V) the score pass uses for max_len
int score_blocks(const ScoreArgs &a, int32_t max_len, int sms, int *V);
// layer groups (grid z) of a score pass over n_elig eligible layers
int score_layer_groups(int n_elig);
cudaError_t launch_entropy_fold(const ScoreArgs &a, int32_t max_len, cudaStream_t st);
cudaError_t launch_vnorm_mean(const ScoreArgs &a, cudaStream_t st);
cudaError_t launch_value_norms(const void *v, const PagedView &pv, const int32_t *len, int32_t batch, int32_t layers,
                               int32_t cap, int dtype, float *vnorm, cudaStream_t st);
cudaError_t launch_ema_update(int32_t rows, int32_t cap, float *ema, const float *score, const int32_t *len,
                              int32_t rows_per_seq, float alpha, int32_t max_len, cudaStream_t st);
cudaError_t launch_select(int32_t rows, int32_t cap, const float *util, const int32_t *len, int32_t rows_per_seq,
                          const int32_t *budget, int32_t *pos, int32_t *keep, int32_t *keep_len, const DeferArgs &df,
                          cudaStream_t st);

struct CompactArgs {
    void *k, *v;
    PagedView pv;
    int32_t batch, layers, rows_per_seq, cap, elem_bytes;
    int32_t mode;               // IKV_COMPACT_*
    int32_t *len, *pos;
    int32_t *start;             // [batch] or null; advanced by the shorter-side mode
    int32_t *done;              // [batch] arrival counters, zero on entry; reset by the last CTA
    float *ema;
    const int32_t *keep, *keep_len;
    int32_t *moves;             // hole-fill: [rows][cap][2] (src, dst), null for stable
    int32_t *n_moves;           // hole-fill: [rows]
    int32_t max_holes;          // > 0: while a sequence's dead slots stay <= max_holes, mark
                                // the evicted slots dead (pos = -1) instead of compacting
    float *vnorm;               // [layers][batch][kv_heads][cap] value-row norms moved with the rows, or null
    int32_t row_by_layer;       // per-layer eviction: keep row b * rows_per_seq + l governs layer l
                                // (all kv heads) and pos row b * rows_per_seq + l
};
cudaError_t launch_compact(const CompactArgs &a, int mode, int sms, cudaStream_t st);

struct AppendArgs {
    void *k, *v;
    PagedView pv;
    int32_t batch, layers, rows_per_seq, cap, elem_bytes;
    const void *k_new, *v_new;  // [layers][batch][kv_heads][D]
    int32_t *len, *pos, *next_pos;
    float *ema;
    int32_t init_mean;
    int32_t dead_slots;         // the mean initialisation skips slots with pos < 0
    int32_t *done;              // [batch] arrival counters, zero on entry; reset by the last CTA
    float *vnorm;               // [layers][batch][kv_heads][cap]: the new row's norm is stored, or null
    // split step: k_new == null makes launch_append do the bookkeeping only and record
    // each sequence's reserved logical slot (-1: no room) in slot[b]; launch_append_rows
    // then writes layer layer0's rows (k_new: [batch][kv_heads][D]) into that slot
    int32_t layer0;
    int32_t *slot;
};
cudaError_t launch_append(const AppendArgs &a, cudaStream_t st);
// rows of layers layer0 .. layer0 + layers - 1 (k_new: [layers][batch][kv_heads][D]) into slot[b]
cudaError_t launch_append_rows(const AppendArgs &a, cudaStream_t st);

// Per-layer eviction (IKV_EVICT_LAYER): a position-indexed state m [batch][pos_cap]
// shared by all layers; layer l's positions in pos row b * layers + l.  Within a step no
// layer's eviction feeds another layer's inputs (each attends its own rows, and a
// layer's update only reads the tokens it held before the step's evictions), so every
// layer's utilities are computed after all attention, by one pass over positions that
// walks the layers in order, and all layers are selected and compacted together.
struct LayerArgs {
    int32_t batch, layers, cap, pos_cap;
    int32_t *len, *next_pos, *pos;
    const int32_t *start;       // [batch] or null
    float *m;                   // [batch][pos_cap] state
    int32_t *inv;               // [batch][layers][pos_cap] workspace: slot of position p in layer l
                                // (stale entries are rejected by checking pos[l][slot] == p)
    uint32_t *live;             // [batch][live_words] workspace: bit p = some layer holds position p
    int32_t live_words;         // ceil(pos_cap / 32)
    float *util;                // [batch][layers][cap] workspace: utilities by slot
    const float *sbuf;          // [batch][n_elig][lstride] pooled scores of the eligible layers
    int32_t lstride, n_elig;
    float alpha;
    int32_t scoring;            // refresh step: fold the eligible layers' scores
    uint32_t elig_bits[kMaxLayers / 32];
    int32_t init_mean;          // begin: new token's state = mean over live positions (else 0)
    int32_t *slot;              // begin: each sequence's reserved slot, -1 if none
};
// live-position bits of the cache before the append (live must be zeroed first), then
// the append bookkeeping; max_len bounds len before the append
cudaError_t launch_layer_begin(const LayerArgs &a, int32_t max_len, cudaStream_t st);
// inverse maps of every layer, then the per-position fold (utilities and final state)
cudaError_t launch_layer_fold(const LayerArgs &a, int32_t max_len, int32_t max_pos, cudaStream_t st);
cudaError_t read_clear_layer_error(unsigned int *v);

// Rank-trace diagnostics (trace.cu)
struct TraceArgs {
    int32_t rows, rows_per_seq, cap;
    const int32_t *len, *pos;       // [batch], [rows][cap] (after the step's eviction)
    const int32_t *keep_raw, *n_raw; // raw top-k slots (ascending) and counts, before eviction
    int32_t *raw_pos;               // [rows][cap] workspace: positions of the raw top-k
    int32_t has_raw;                // refresh step: R_t exists
    int32_t *raw_top, *ema_top, *n_top, *counts;
};
// raw_pos[r][j] = pos[r][keep_raw[r][j]] (before the eviction moves pos)
cudaError_t launch_trace_gather(const TraceArgs &a, int32_t max_len, cudaStream_t st);
cudaError_t launch_trace(const TraceArgs &a, cudaStream_t st);
cudaError_t read_clear_trace_error(unsigned int *v);
// reads and clears the append kernel's device error word (bit 0: no free slot)
cudaError_t read_clear_append_error(unsigned int *v);

}  // namespace ikv
