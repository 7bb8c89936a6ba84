/*
 * epikv.h -- C ABI of the EpiKV eviction hot path for NVIDIA GB300 (sm_103a).
 *
 * EpiKV ("Epiphany-Aware KV Cache Eviction Without the Attention Matrix")
 * scores every generated token once, from quantities the forward pass
 * already produces, and keeps the K best tokens of each sequence's KV cache:
 *
 *   score   Band-z ("EpiKV"): g_l(t) = ||h_l(t) - h_l(t-1)||_2 per band layer
 *           (Sec. 3.2, Eq. 1), a causal rolling z-score per layer (Eq. 3),
 *           Band A mean minus Band B mean (Fig. 1).
 *           Lag-KV: each token's K and V vectors normalised by the previous
 *           chunk's per-channel range, variance over the head dimension, key
 *           + value, mean over (layer, head), rolling mean (Sec. 3.3).
 *   select  keep all prefill tokens and the last min(128, K/4) tokens, and
 *           give the rest of the budget K to the highest-scoring tokens
 *           (Sec. 3.1, Sec. 3.3, App. D).
 *   compact rewrite every layer's and head's K/V rows to the kept set, in
 *           token order (App. H).
 *
 * Conventions shared by every call
 *   - Ownership: the caller owns every buffer (the workspace, hidden rows,
 *     the K/V pool, block tables, outputs).  The library never allocates
 *     device memory; epikv_init allocates only its small host-side context.
 *   - Asynchrony: every call except epikv_get_error, epikv_get_stats,
 *     epikv_read_slots and epikv_read_layer_slots only enqueues work on the
 *     given stream and returns (no synchronisation, no allocation), so a
 *     whole decode step can be captured once in a CUDA graph and replayed.
 *     Calls on one context must be ordered on one stream.
 *   - Host validation failures return EPIKV_EINVAL and enqueue nothing.
 *   - Device-side anomalies (an index out of range, a batch larger than
 *     declared, a kept list that is not strictly increasing) never trap:
 *     the kernel records a code in the context's sticky error word and
 *     skips the offending work.  epikv_get_error returns and clears it.
 *   - bf16 data; K/V rows of one token and layer are H*d contiguous
 *     elements (head-major, channel-minor); all pointers 16-byte aligned.
 *   - A sequence id appears at most once in one call's batch.
 *   - A call's kernels are launched with programmatic dependent launch
 *     among themselves (each waits for its predecessor's results before it
 *     reads anything); against the caller's own work on the stream the
 *     order is plain stream order, except that a caller kernel itself
 *     launched with programmatic dependent launch right after a call must,
 *     as with any such launch, wait for its predecessor
 *     (cudaGridDependencySynchronize) before reading the call's results.
 */
#ifndef EPIKV_H_
#define EPIKV_H_

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  EPIKV_OK = 0,
  EPIKV_EINVAL = 1,   /* invalid argument or configuration; nothing enqueued */
  EPIKV_ECUDA = 2,    /* a CUDA runtime call or kernel launch failed */
  EPIKV_EDEVICE = 3,  /* the device error word was set (see epikv_device_error) */
} epikv_status;

/* Codes a kernel writes into the sticky device error word (first one wins). */
typedef enum {
  EPIKV_DEV_OK = 0,
  EPIKV_DEV_BATCH = 1,      /* n_new < 0 or > max_new, or seq id out of range */
  EPIKV_DEV_CAPACITY = 2,   /* n_cache + n_new would exceed max_cache_tokens */
  EPIKV_DEV_SLOT = 3,       /* a slot or block index outside the KV view */
  EPIKV_DEV_KEPT = 4,       /* kept list not strictly increasing / out of range */
  EPIKV_DEV_BUDGET = 5,     /* budget K < 1 or > max_cache_tokens */
  EPIKV_DEV_TIMEOUT = 6,    /* a bounded wait inside a kernel gave up */
} epikv_device_error;

/* Score kinds (bit mask in epikv_config.score_kinds, one value as policy).
 *   BANDZ   EpiKV: Band A mean - Band B mean of rolling z-scores of g (Eq. 3)
 *   LAGKV   Lag-KV: lag-normalised key + value head variance (Sec. 3.3)
 *   HSVAR   HS-variance: Band A mean - Band B mean of rolling means of g (Eq. 2)
 *   KVKEY   KV-key: rolling mean of the stored keys' head variance (Sec. 3.3)
 *   KVVAL   KV-val: the same for the values (Sec. 3.3)
 *   LAGKEY  lag-kv-key: Lag-KV's key term only (Tab. "acc-math" rows)
 * The band kinds use z_window as their window; the K/V kinds lag_window. */
enum {
  EPIKV_SCORE_BANDZ = 1,
  EPIKV_SCORE_LAGKV = 2,
  EPIKV_SCORE_HSVAR = 4,
  EPIKV_SCORE_KVKEY = 8,
  EPIKV_SCORE_KVVAL = 16,
  EPIKV_SCORE_LAGKEY = 32,
};

/* KV cache layouts. */
enum { EPIKV_LAYOUT_CONTIGUOUS = 0, EPIKV_LAYOUT_PAGED = 1 };

typedef struct {
  int32_t max_seqs;         /* sequence ids are 0..max_seqs-1 */
  int32_t max_cache_tokens; /* cache slots per sequence (T_cap) */
  int32_t max_new_tokens;   /* new tokens per sequence per score update, max */
  int32_t num_layers;       /* L: layers of the K/V cache */
  int32_t num_kv_heads;     /* H */
  int32_t head_dim;         /* d: a power of two in [8, 256]; H*d/8 <= 256 */
  int32_t hidden;           /* D: hidden size, a multiple of 8, <= 8192 */
  int32_t n_band_a;         /* Band A layers passed per update (Sec. 3.2: 7..13) */
  int32_t n_band_b;         /* Band B layers (Sec. 3.2: 18..25); A+B <= 32 */
  int32_t z_window;         /* w of Eq. 2 and 3 (paper: 64), 1..1024 */
  float z_eps;              /* epsilon of Eq. 3 (1e-6) */
  int32_t lag;              /* Lag-KV chunk length (16), >= 1 */
  float lag_eps;            /* epsilon of the range normalisation (1e-6) */
  int32_t lag_window;       /* rolling-mean window of the K/V scores (64), 1..1024 */
  int32_t recency_cap;      /* recency window R = min(recency_cap, K/4) (App. D: 128) */
  int32_t score_kinds;      /* EPIKV_SCORE_* mask (1..63) computed by every update */
  int32_t select_chunk;     /* C, 0..65536 (0 reads as 1).  1: the paper's token-level top-K.
                             * C > 1: chunk-level selection, which the paper names as future
                             * work (Sec. 5, after ChunkKV's contiguous chunks, Sec. 2): the
                             * candidates fall into fixed position chunks floor(pos / C), a
                             * chunk scores the fp32 mean of its candidate members' scores
                             * (summed in slot order), and whole chunks fill the candidate
                             * budget in rank order (NaN lowest, ties to the earlier chunk);
                             * the first chunk that does not fit keeps its lowest slots. */
  int32_t layer_budgets;    /* 0: one budget per sequence (the paper's method).  1: one budget
                             * per (sequence, layer), which the paper names as future work
                             * (Sec. 5, after PyramidKV's per-layer allocation, Sec. 2): layer
                             * l keeps its own cache of n_l slots and evicts it with its own
                             * budget K_l at the sequence's events; every layer keeps the
                             * prefill and one shared recency window R = min(recency_cap,
                             * K_min/4) (shrunk to K_min - P), K_min the smallest budget.
                             * Needs num_layers <= 64 and select_chunk <= 1.  In this mode
                             * the per-entry budget, kept and length arrays of epikv_select,
                             * epikv_compact and epikv_step gain a layer dimension (see
                             * there), "n_cache" is the largest layer's length, and the new
                             * K/V rows of an update go to slots n_l .. n_l+n_new-1 of each
                             * layer. */
} epikv_config;

/* New hidden-state rows of one update call (Sec. 3.1: the per-layer hidden
 * states of the standard output_hidden_states interface).  band_rows[i] is a
 * device pointer to bf16 rows [total_new][row_stride] of band layer i (the
 * n_band_a Band A layers first, then the Band B layers); batch entry b owns
 * rows cu_new[b] .. cu_new[b+1]-1, in position order. */
typedef struct {
  const void* band_rows[32];
  int64_t row_stride;       /* elements between consecutive rows (>= hidden) */
} epikv_hidden_view;

/* The K/V cache (Sec. 3.1: 2*L*H*d scalars per token).  Element offsets:
 *   contiguous: layer*stride_layer + seq*stride_seq + slot*stride_token
 *   paged:      layer*stride_layer + block_table[layer*stride_table_layer +
 *               seq*max_blocks_per_seq + slot/block_size]*stride_block +
 *               (slot%block_size)*stride_token
 * The same offsets address k and v.  stride_table_layer = 0 shares one block
 * table among the layers; with per-layer budgets, stride_layer = 0 and one
 * table per layer describe a single pool of blocks in which every (layer,
 * sequence) owns its own blocks, so each layer's memory follows its own
 * budget.  The caller keeps distinct (layer, sequence) block lists disjoint. */
typedef struct {
  void* k;
  void* v;
  int32_t layout;               /* EPIKV_LAYOUT_* */
  int64_t stride_layer;
  int64_t stride_seq;           /* contiguous only */
  int64_t stride_block;         /* paged only */
  int64_t stride_token;         /* usually H*d */
  const int32_t* block_table;   /* paged only: device int32 [max_seqs][max_blocks_per_seq] */
  int32_t max_blocks_per_seq;   /* paged only */
  int32_t block_size;           /* paged only: tokens per block */
  int32_t num_blocks;           /* paged only: pool size, for bounds checks */
  int64_t stride_table_layer;   /* paged only: elements between consecutive layers' block
                                 * tables (0: one table for every layer) */
} epikv_kv_view;

typedef struct {
  unsigned long long tokens_scored;  /* new tokens accepted by score updates */
  unsigned long long evictions;      /* (sequence, event) pairs that evicted */
  unsigned long long rows_moved;     /* kept tokens whose slot changed (largest layer) */
  unsigned long long layer_rows_moved; /* (layer, kept token) pairs whose slot changed */
} epikv_stats;

typedef struct epikv_ctx epikv_ctx;

/* Bytes of device workspace epikv_init needs for cfg (0 if cfg is invalid):
 * the per-sequence state (counters, frozen scores and positions per slot,
 * score rings, Lag-KV chunk ranges, kept lists) plus a fixed compaction stash
 * of 512 x min(128, max_cache_tokens) K/V rows of one layer (128 MiB at
 * num_kv_heads * head_dim = 1024). */
size_t epikv_workspace_bytes(const epikv_config* cfg);

/* Create a context over a caller-allocated device workspace of at least
 * epikv_workspace_bytes(cfg) bytes (256-byte aligned), zero it on `stream`
 * and reset every sequence.  *out receives a host-side handle. */
epikv_status epikv_init(epikv_ctx** out, const epikv_config* cfg, void* d_workspace,
                        size_t workspace_bytes, cudaStream_t stream);

/* Start sequence `seq` afresh: empty cache, next position 0, `prefill_len`
 * leading tokens that are never evicted (App. D: all prefill kept), and the
 * score kind that drives its selection (`policy`, one EPIKV_SCORE_* value
 * that is in cfg.score_kinds). */
epikv_status epikv_seq_reset(epikv_ctx* ctx, int32_t seq, int32_t prefill_len, int32_t policy,
                             cudaStream_t stream);

/* Score the new tokens of a batch and append them to each sequence's slots.
 *   d_seq_ids [n_seq]   device: sequence id of each batch entry
 *   d_cu_new  [n_seq+1] device: prefix offsets of the new tokens per entry
 *                       (d_cu_new[0] = 0, non-decreasing)
 *   max_new             host: an upper bound of every entry's new tokens
 *                       (<= cfg.max_new_tokens; sizes the grid)
 *   hidden              band rows of the new tokens (needed for BANDZ, HSVAR)
 *   kv                  the cache; the new tokens' K/V rows must already be
 *                       in slots n_cache .. n_cache+n_new-1 (needed for the
 *                       K/V kinds)
 * Each token's score is computed once, causally, and frozen (Sec. 3.3). */
epikv_status epikv_score_update(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids,
                                const int32_t* d_cu_new, int32_t max_new,
                                const epikv_hidden_view* hidden, const epikv_kv_view* kv,
                                cudaStream_t stream);

/* Choose the kept tokens of each batch entry (Sec. 3.1, App. D).
 *   d_budget  [n_seq] device: budget K per entry
 *   d_trigger [n_seq] device or NULL: evict only if n_cache > trigger
 *             (NULL: evict whenever n_cache > K)
 *   d_kept    device int32 [n_seq][kept_stride]: ascending kept slots,
 *             written only for entries that evict
 *   d_n_kept  device int32 [n_seq]: the cache length after the call
 * With cfg.layer_budgets = 1: d_budget is [n_seq][num_layers] (K_l of each
 * layer), an entry evicts if n_cache (its largest layer) exceeds the trigger
 * (NULL: the largest K_l) and the smallest K_l; d_kept is
 * [n_seq][num_layers][kept_stride], each layer's kept slots in its own slot
 * numbering, and d_n_kept is [n_seq][num_layers]; kept_stride must be at
 * least max(K_max, prefill).  A sequence's layer budgets must stay the same
 * from one epikv_seq_reset to the next: the library keeps one ranking for
 * all layers, which is exact because fixed budgets keep the layers' caches
 * nested; a change that would break the nesting is reported as
 * EPIKV_DEV_KEPT.
 * Ties between equal scores go to the lower slot, NaN ranks lowest.  The
 * call commits the eviction to the context's slot metadata (scores and
 * positions move with their tokens); the caller must apply epikv_compact
 * with the same kept lists, once, before the next score update. */
epikv_status epikv_select(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids,
                          const int32_t* d_budget, const int32_t* d_trigger, int32_t* d_kept,
                          int32_t kept_stride, int32_t* d_n_kept, cudaStream_t stream);

/* Move every layer's K and V rows of the entries that evicted in the
 * preceding epikv_select to their kept slots, in order, in place (App. H).
 * Rows before the first evicted slot are not touched.  d_kept has the layout
 * epikv_select wrote (per layer with cfg.layer_budgets = 1).  An eviction is
 * applied once: calling epikv_compact again, or with no eviction selected
 * since the last score update, moves nothing; a score update that finds an
 * eviction selected but not yet compacted reports EPIKV_DEV_KEPT. */
epikv_status epikv_compact(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids,
                           const int32_t* d_kept, int32_t kept_stride, const epikv_kv_view* kv,
                           cudaStream_t stream);

/* One decode step: epikv_score_update, then a device-side trigger
 * (evict entries with n_cache > trigger), epikv_select into the context's
 * own kept buffer and epikv_compact -- without any host synchronisation.
 *   d_n_cache_out [n_seq] device or NULL: each entry's cache length after
 *                 the step (a paged caller frees blocks past it);
 *                 [n_seq][num_layers], every layer's length, with
 *                 cfg.layer_budgets = 1 (d_budget as in epikv_select). */
epikv_status epikv_step(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids,
                        const int32_t* d_cu_new, int32_t max_new, const int32_t* d_budget,
                        const int32_t* d_trigger, const epikv_hidden_view* hidden,
                        const epikv_kv_view* kv, int32_t* d_n_cache_out, cudaStream_t stream);

/* Record events[0..3] on the stream at the phase boundaries of every later
 * epikv_step (before scoring, before select, before compact, after compact);
 * NULL stops it.  The events are the caller's. */
epikv_status epikv_set_phase_events(epikv_ctx* ctx, const cudaEvent_t* events);

/* Per-kernel timing for measurement.  From this call on, every kernel that an
 * entry point of `ctx` launches (epikv_score_update, epikv_select,
 * epikv_compact, epikv_step) is bracketed on its stream by two of the
 * caller's events -- events[2k] before and events[2k+1] after the k-th such
 * kernel -- and h_names[k] receives its name as the CUDA runtime reports it
 * (storage owned by the runtime), for at most n_kernels kernels; later ones
 * are not recorded.  Both arrays are the caller's and must stay valid until
 * the next call.  An event recorded between two kernels also ends the early
 * launch of the second (programmatic dependent launch), so the kernels then
 * run strictly one after another.  events == NULL stops it and, if h_used is
 * not NULL, stores how many kernels were recorded.  Not thread safe with
 * respect to other calls on the same context. */
epikv_status epikv_set_kernel_events(epikv_ctx* ctx, const cudaEvent_t* events, int32_t n_kernels,
                                     const char** h_names, int32_t* h_used);

/* Debug/test read-back (synchronises): the cache length, positions and
 * scores of kind `kind` of `seq`'s slots; at most `cap` entries copied. */
epikv_status epikv_read_slots(epikv_ctx* ctx, int32_t seq, int32_t kind, float* h_score,
                              int32_t* h_pos, int32_t cap, int32_t* h_n);

/* Debug/test read-back (synchronises), cfg.layer_budgets = 1 only: the
 * length n_l of layer `layer` of `seq` and the positions its slots hold, at
 * most `cap` of them. */
epikv_status epikv_read_layer_slots(epikv_ctx* ctx, int32_t seq, int32_t layer, int32_t* h_pos,
                                    int32_t cap, int32_t* h_n);

/* Synchronise the last stream used and return the cumulative counters. */
epikv_status epikv_get_stats(epikv_ctx* ctx, epikv_stats* out);

/* Synchronise; EPIKV_EDEVICE if the device error word is set, with its code
 * in *code (may be NULL); the word is cleared. */
epikv_status epikv_get_error(epikv_ctx* ctx, int32_t* code);

/* Lag-KV scores of positions 0..n-1 of one sequence, in one call that needs
 * no context and no device memory beyond its arguments.  The paper has no
 * counterpart to this entry point: it is for callers that cannot allocate
 * device memory -- a plugin inside an application whose memory pool owns the
 * whole GPU, an embedded caller without a device allocator, or a loop that
 * must never block on cudaMalloc -- and so cannot create the workspace that
 * epikv_init needs.  Its scores agree, to fp32 rounding, with the ones
 * epikv_score_update gives for the same tokens of a fresh sequence.
 *   kv         the caller's cache; slots 0..n-1 of `seq` hold positions 0..n-1
 *   L, H, d    layers, KV heads, head dim (d a power of two in [8, 256],
 *              H <= 32, H*d/8 <= 256)
 *   lag, lag_eps, window   as in epikv_config
 *   d_scores   device float [n]: the output
 * Working memory is a fixed 2 MiB array inside the library (every GPU that
 * loads the library holds it until the process exits), so n * 2 * L must not
 * exceed 524,288 (n <= 8,192 at L = 32): larger requests return EPIKV_EINVAL
 * and launch nothing.  The first call in each CUDA context looks the array's
 * address up (with that context current) and remembers it under the
 * context's unique id, so a context created again after cudaDeviceReset gets
 * a fresh lookup; make the first call in a context before any stream
 * capture.  All calls share the array: calls that overlap on the GPU
 * (unordered streams) race and must be avoided; calls ordered on one stream
 * are independent.  Slots the view does not map (a negative or out-of-range
 * block-table entry) are read as zero rows and are not reported.  A CUDA
 * error already pending on the calling thread is returned as EPIKV_ECUDA
 * before anything is launched, and left in place for its owner. */
epikv_status epikv_lagkv_score_noalloc(const epikv_kv_view* kv, int32_t seq, int32_t n,
                                       int32_t num_layers, int32_t num_kv_heads, int32_t head_dim,
                                       int32_t lag, float lag_eps, int32_t window, float* d_scores,
                                       cudaStream_t stream);

void epikv_destroy(epikv_ctx* ctx);
const char* epikv_status_string(epikv_status s);

#ifdef __cplusplus
}
#endif
#endif /* EPIKV_H_ */
