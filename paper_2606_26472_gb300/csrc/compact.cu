// In-place, order-preserving K/V compaction to the kept set (App. H).
//
// For every sequence that evicted in the last selection and every
// (layer, K|V, head group) stream: row i <- row kept[i] for i from the first
// evicted slot to the new cache length.  Rows are moved with 1-D TMA bulk
// copies global -> shared -> global (cp.async.bulk + mbarrier), no cluster
// multicast.  A persistent grid of one-warp CTAs walks its streams' batches
// through a ring of shared-memory stages: while batch k is stored, batches
// k+1 .. k+S-1 are loading.
//
// In-place safety without any inter-CTA wait: streams are disjoint bytes;
// inside a CTA's rows of a stream kept[i] >= i and rows are processed in
// increasing i, so a load (slot kept[i] >= i) never reads a slot that an
// earlier store has written, and a later store to a slot some earlier batch
// still had to read is issued only after that batch's loads completed.  With
// per-stream units one CTA owns each stream; the balanced split below cuts
// streams between CTAs and covers the reads across a cut with a stash.
//
// Under per-layer budgets (kLayers) each (sequence, layer) has its own kept
// list, first moved slot and length; the streams and the copy are unchanged.
// The balanced split then runs over (sequence, layer) pairs of two streams
// each.  Without it the streams differ in length (a layer's rows follow its
// budget), so the CTAs take units from a shared counter instead of a fixed
// stride, in layer-major order: with budgets that fall with depth, larger
// streams come first and the greedy assignment ends nearly level.
//
// Balanced split: the moved rows of all evicting streams,
// laid end to end, are cut into one equal chunk per CTA, so one evicting
// sequence still covers the whole grid and no CTA carries a longer share.
// A chunk that ends inside a stream at slot a still reads, for its last rows,
// sources in [a, n_new) that later chunks overwrite.  compact_stash_kernel
// copies those rows aside before the compaction starts, and the chunk reads
// them there.  They are a suffix of the chunk's rows in that stream, no
// longer than the chunk nor than the eviction's largest shift
// kept[n-1] - (n-1); when both bounds exceed the stash, the per-stream units
// above are used instead.
//
// A selection's eviction is compacted once: compact_consumed_kernel, launched
// after the copy, sets each sequence's first moved slot to its length, so
// another compaction before the next selection moves nothing.
#include "common.cuh"
#include "kernels.h"

namespace epikv {

#ifndef EPIKV_COMPACT_STAGE_BYTES
#define EPIKV_COMPACT_STAGE_BYTES 16384
#endif
#ifndef EPIKV_COMPACT_STAGES
#define EPIKV_COMPACT_STAGES 4
#endif
#ifndef EPIKV_COMPACT_CTAS_PER_SM
#define EPIKV_COMPACT_CTAS_PER_SM 2  // more CTAs per SM overload the memory system (measured)
#endif
#ifndef EPIKV_COMPACT_ORDER
#define EPIKV_COMPACT_ORDER 0  // 0: units sequence-major, 1: layer-major
#endif
#ifndef EPIKV_COMPACT_HEAD_SPLIT
#define EPIKV_COMPACT_HEAD_SPLIT 0  // 0: chosen on the device to fill the grid
#endif
constexpr int kStageBytes = EPIKV_COMPACT_STAGE_BYTES;
constexpr int kStages = EPIKV_COMPACT_STAGES;
constexpr int kMaxRowsPerLane = 4;
constexpr int kMaxRPB = 32 * kMaxRowsPerLane;
constexpr uint64_t kWaitNs = 2000000000ull;   // 2 s: far beyond any real copy
constexpr uint64_t kDrainNs = 100000000ull;   // 0.1 s per stage after a timeout

#ifndef EPIKV_COMPACT_BALANCED
#define EPIKV_COMPACT_BALANCED 1  // 0: per-stream units only
#endif
#ifndef EPIKV_COMPACT_STAGED_BLOCKS
#define EPIKV_COMPACT_STAGED_BLOCKS 1024  // block-table entries kept in shared memory (larger tables: global reads)
#endif
constexpr int kStagedBlocks = EPIKV_COMPACT_STAGED_BLOCKS;

constexpr int kStashThreads = 512;
constexpr int kStashUnroll = 4;

// The balanced split's row space is made of pairs: under token budgets one
// per evicting entry, with its 2L streams; under per-layer budgets one per
// (evicting entry, layer), with that layer's K and V streams, at most
// kMaxLayerPairs of them (more: per-stream units).
// Per-layer budgets, 32 layers, 8,192-slot caches evicting 128 slots per
// step (compaction ms, balanced / per-stream units): 1 sequence 0.35 / 1.09,
// 2 sequences 0.68 / 1.24, 8 sequences 2.59 / 2.68, 32 sequences 10.18 /
// 9.95.  So the balanced split takes at most 256 (entry, layer) pairs.
#ifndef EPIKV_COMPACT_LAYER_PAIRS
#define EPIKV_COMPACT_LAYER_PAIRS 256
#endif
constexpr int kMaxLayerPairs = EPIKV_COMPACT_LAYER_PAIRS;
__host__ __device__ inline int list_ints(int n_seq) { return (n_seq + 31) / 32 * 32; }
__host__ __device__ inline int pairs_cap(int n_seq, int L, bool layers) {
  return layers ? (n_seq * L < kMaxLayerPairs ? n_seq * L : kMaxLayerPairs) : n_seq;
}
__host__ __device__ inline int pre_entries(int cap) { return (cap + 32) / 32 * 32; }

// The batch entries that evicted, in batch order, into list; with pre, the
// prefix sums of their moved rows per stream (pre[k] = rows of entries
// before the k-th).  One warp; every CTA of both kernels builds the same.
// Every entry's moved rows are loaded first (list holds them, list_ints(n_seq)
// >= n_seq words), all loads in flight together, then scanned in place.
__device__ int evicting_entries(const DevState& st, const Dims& dm, const int32_t* __restrict__ seq_ids,
                                int n_seq, int* list, int64_t* pre, int lane) {
#pragma unroll 4
  for (int b = lane; b < n_seq; b += 32) {
    const int seq = seq_ids[b];
    list[b] = (seq >= 0 && seq < dm.S) ? st.n_cache[seq] - st.first_changed[seq] : 0;
  }
  __syncwarp();
  int n_ev = 0;
  int64_t acc = 0;
  for (int base = 0; base < n_seq; base += 32) {
    const int b = base + lane;
    const int len = b < n_seq ? list[b] : 0;
    __syncwarp();  // the chunk's lengths are read before any of its entries is written
    const bool ev = len > 0;
    const unsigned m = __ballot_sync(0xffffffffu, ev);
    int incl = ev ? len : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (ev) {
      const int k = n_ev + __popc(m & ((1u << lane) - 1u));
      list[k] = b;   // k <= b: an entry already read
      if (pre) pre[k + 1] = acc + incl;
    }
    acc += __shfl_sync(0xffffffffu, incl, 31);
    n_ev += __popc(m);
    __syncwarp();
  }
  if (pre && lane == 0) pre[0] = 0;
  __syncwarp();
  return n_ev;
}

// Per-layer budgets: the prefix sums over the (entry, layer) pairs of their
// moved rows per stream (pre[k] = rows of the pairs before the k-th, pair k
// = entry k / L, layer k % L).  One warp; returns the pairs' total.
__device__ int64_t layer_pairs(const DevState& st, const Dims& dm, const int32_t* __restrict__ seq_ids,
                               const int* list, int n_ev, int64_t* pre, int lane) {
  const int np = n_ev * dm.L;
  // every pair's rows first (independent loads, several in flight), then the scan
#pragma unroll 4
  for (int k = lane; k < np; k += 32) {
    const int i = seq_ids[list[k / dm.L]] * dm.L + k % dm.L;
    pre[k + 1] = max(0, st.n_layer[i] - st.lfirst[i]);
  }
  __syncwarp();
  int64_t acc = 0;
  for (int base = 0; base < np; base += 32) {
    const int k = base + lane;
    const int len = k < np ? (int)pre[k + 1] : 0;
    int incl = len;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (k < np) pre[k + 1] = acc + incl;
    acc += __shfl_sync(0xffffffffu, incl, 31);
  }
  if (lane == 0) pre[0] = 0;
  __syncwarp();
  return acc;
}

// One pair's stream q (token budgets: layer * 2 + K|V; per-layer budgets:
// K|V): its entry, sequence, layer, first moved row, new length and kept list.
struct PairAt {
  int b, seq, layer, kvk, first, n_new;
  const int32_t* kl;
};
__device__ __forceinline__ PairAt pair_at(const DevState& st, const Dims& dm, const int32_t* __restrict__ seq_ids,
                                          const int* list, const int32_t* __restrict__ kept, int kept_stride,
                                          bool layers, int p, int q) {
  PairAt a;
  a.b = list[layers ? p / dm.L : p];
  a.seq = seq_ids[a.b];
  if (layers) {
    a.layer = p % dm.L;
    a.kvk = q;
    const int i = a.seq * dm.L + a.layer;
    a.first = st.lfirst[i];
    a.n_new = st.n_layer[i];
    a.kl = kept + ((size_t)a.b * dm.L + a.layer) * kept_stride;
  } else {
    a.layer = q >> 1;
    a.kvk = q & 1;
    a.first = st.first_changed[a.seq];
    a.n_new = st.n_cache[a.seq];
    a.kl = kept + (size_t)a.b * kept_stride;
  }
  return a;
}

// Whether the balanced split applies: a grid within the stash's CTAs, under
// per-layer budgets no more pairs than kMaxLayerPairs, and a bound on the
// rows of a chunk whose sources lie in later chunks' regions -- a suffix of
// the chunk's last stream segment, no longer than the segment (so than the
// chunk, ceil(total / grid) rows) nor than the largest shift
// kept[n-1] - (n-1) of any pair -- within one CTA's stash.  total = moved
// rows of all streams.
__device__ bool balanced_split(const DevState& st, const Dims& dm, const int32_t* __restrict__ seq_ids,
                               const int* list, int n_ev, const int32_t* __restrict__ kept, int kept_stride,
                               bool layers, int n_pairs, int64_t total, int lane) {
  if (!EPIKV_COMPACT_BALANCED || gridDim.x > kMaxStashCtas) return false;
  if (layers && n_pairs > kMaxLayerPairs) return false;
  if ((total + gridDim.x - 1) / gridDim.x <= dm.stash_rows) return true;
  bool ok = true;
#pragma unroll 4
  for (int k = lane; k < n_pairs; k += 32) {
    const PairAt a = pair_at(st, dm, seq_ids, list, kept, kept_stride, layers, k, 0);
    if (a.n_new > a.first) ok &= __ldg(a.kl + a.n_new - 1) - (a.n_new - 1) <= dm.stash_rows;
  }
  return __all_sync(0xffffffffu, ok);
}

// Entry e, stream q (layer * 2 + K|V) and row r (from the entry's first
// moved slot) of row o of the balanced row space.
__device__ __forceinline__ void locate_row(const int64_t* pre, int n_ev, int upe, int64_t o, int& e, int& q,
                                           int64_t& r) {
  int lo = 0, hi = n_ev - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pre[mid] * upe <= o) lo = mid;
    else hi = mid - 1;
  }
  e = lo;
  const int64_t len = pre[e + 1] - pre[e];
  const int64_t rel = o - pre[e] * upe;
  q = (int)(rel / len);
  r = rel - (int64_t)q * len;
}

struct Cursor {
  int u;      // unit index (this CTA strides by gridDim.x); balanced: 0 while rows remain
  int i;      // next row of the unit
  int end;    // row past the last of the unit
  int b, seq, layer, kvk, hg;
  int stash_at;   // balanced: sources in [stash_at, n_new) are read from the next chunk's stash
  int n_new;      // balanced: the sequence's length after the eviction
  int row0;       // balanced: the row whose source is the stash's first row
  int64_t o_end;  // balanced: row `end` in the balanced row space
};

// kSplit: the balanced split is compiled in (token budgets always; per-layer
// budgets when the batch has at most kMaxLayerPairs (entry, layer) pairs --
// the instance for larger batches keeps the per-stream units' code alone,
// which measured 6 % faster there than with the split's code beside it).
template <bool kLayers, bool kSplit>
__global__ void __launch_bounds__(32) compact_kernel(DevState st, Dims dm, KvDev kv,
                                                     const int32_t* __restrict__ seq_ids, int n_seq,
                                                     const int32_t* __restrict__ kept, int kept_stride) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t full[kStages];
  __shared__ char* dptr[kStages][kMaxRPB];
  __shared__ int stage_rows[kStages];
  int* list = reinterpret_cast<int*>(smem + kStages * kStageBytes);
  int64_t* pre = reinterpret_cast<int64_t*>(list + list_ints(n_seq));
  // the current sequence's block table
  int* bt_s = reinterpret_cast<int*>(pre + pre_entries(pairs_cap(n_seq, dm.L, kLayers)));
  const int lane = threadIdx.x;

  // ---- the batch entries that evicted (every CTA builds the same list)
  const int n_ev = evicting_entries(st, dm, seq_ids, n_seq, list, kLayers ? nullptr : pre, lane);
  if (n_ev == 0) return;
  // ---- the balanced split's pairs and their rows
  const int n_pairs = kLayers ? n_ev * dm.L : n_ev;
  const int sp = kLayers ? 2 : 2 * dm.L;  // streams per pair
  int64_t pair_rows = 0;
  bool balanced = false;
  if constexpr (kSplit) {
    if (!kLayers) pair_rows = pre[n_ev];
    else if (n_pairs <= kMaxLayerPairs) pair_rows = layer_pairs(st, dm, seq_ids, list, n_ev, pre, lane);
    balanced = (!kLayers || n_pairs <= kMaxLayerPairs) &&
               balanced_split(st, dm, seq_ids, list, n_ev, kept, kept_stride, kLayers, n_pairs, pair_rows * sp,
                              lane);
  }

  // ---- per-stream units only: whole token rows unless too few streams
  // evict to give every CTA one (small TMA copies cost much more per byte
  // than a tail)
  const int G = gridDim.x;
  int hs = 1;
  if (!balanced) {
#if EPIKV_COMPACT_HEAD_SPLIT > 0
    if (dm.H % EPIKV_COMPACT_HEAD_SPLIT == 0) hs = EPIKV_COMPACT_HEAD_SPLIT;
#else
    while ((long)n_ev * 2 * dm.L * hs < G && dm.H % (2 * hs) == 0 && (dm.H / (2 * hs)) * dm.d * 2 >= 256) hs *= 2;
#endif
  }
  const int rb = (dm.H / hs) * dm.d * 2;               // bytes per row piece
  const int64_t piece_elems = (int64_t)(dm.H / hs) * dm.d;
  const int rpb = min(kStageBytes / rb, kMaxRPB);      // rows per batch
  const int upe = 2 * dm.L * hs;
  const int units = balanced ? 1 : n_ev * upe;
  // balanced: this CTA's chunk [o_begin, o_stop) of the row space
  int64_t o_begin = 0, o_stop = 0;
  if (balanced) {
    const int64_t total = pair_rows * sp;
    o_begin = (int64_t)blockIdx.x * total / G;
    o_stop = (int64_t)(blockIdx.x + 1) * total / G;
  }
  const bool paged = kv.layout == EPIKV_LAYOUT_PAGED;
  const bool bt_in_smem = paged && kv.max_blocks <= kStagedBlocks;

  if (lane == 0) {
    for (int s = 0; s < kStages; ++s) mbar_init(&full[s], 1);
    fence_barrier_init();
    fence_proxy_async_smem();
  }
  __syncwarp();

  // the next unit of this CTA: a fixed stride, or the shared counter (kLayers)
  auto next_unit = [&](int u) -> int {
    if (!kLayers) return u + G;
    int v = 0;
    if (lane == 0) v = (int)atomicAdd(st.work, 1u);
    return __shfl_sync(0xffffffffu, v, 0);
  };
  auto load_unit = [&](Cursor& c) {
    while (c.u < units) {
      int e, rem;
      if (kLayers || EPIKV_COMPACT_ORDER == 1) {
        e = c.u % n_ev;
        rem = c.u / n_ev;
      } else {
        e = c.u / upe;
        rem = c.u % upe;
      }
      c.layer = rem / (2 * hs);
      c.kvk = (rem / hs) & 1;
      c.hg = rem % hs;
      c.b = list[e];
      c.seq = seq_ids[c.b];
      if (kLayers) {
        c.i = st.lfirst[c.seq * dm.L + c.layer];
        c.end = st.n_layer[c.seq * dm.L + c.layer];
      } else {
        c.i = st.first_changed[c.seq];
        c.end = st.n_cache[c.seq];
      }
      c.stash_at = INT_MAX;
      if (c.i < c.end) return;
      c.u = next_unit(c.u);
    }
  };
  // balanced: the stream segment holding row o of the chunk
  auto open_at = [&](Cursor& c, int64_t o) {
    int p, q;
    int64_t r;
    locate_row(pre, n_pairs, sp, o, p, q, r);
    const PairAt a = pair_at(st, dm, seq_ids, list, kept, kept_stride, kLayers, p, q);
    c.b = a.b;
    c.seq = a.seq;
    c.layer = a.layer;
    c.kvk = a.kvk;
    c.hg = 0;
    const int64_t rest = pre[p + 1] - pre[p] - r;       // rows of the stream from o on
    c.i = a.first + (int)r;
    if (o_stop - o < rest) {                             // the chunk ends inside this stream
      c.end = c.i + (int)(o_stop - o);
      c.stash_at = c.end;
      c.n_new = a.n_new;
      c.row0 = st.stash_row0[blockIdx.x + 1];            // written by compact_stash_kernel
    } else {
      c.end = c.i + (int)rest;
      c.stash_at = INT_MAX;
    }
    c.o_end = o + (c.end - c.i);
  };
  auto advance = [&](Cursor& c) {
    c.i += rpb;
    if (c.i >= c.end) {
      if (balanced) {
        if (c.o_end < o_stop) open_at(c, c.o_end);
        else c.u = units;
      } else {
        c.u = next_unit(c.u);
        load_unit(c);
      }
    }
  };
  // kept slots of the batch at c, one load per row, issued early and used later
  auto prefetch = [&](const Cursor& c, int (&pk)[kMaxRowsPerLane]) {
    if (c.u >= units) return;
    const int nrows = min(rpb, c.end - c.i);
    const int32_t* kl = kept + (kLayers ? (size_t)c.b * dm.L + c.layer : (size_t)c.b) * kept_stride + c.i;
#pragma unroll
    for (int j = 0; j < kMaxRowsPerLane; ++j) {
      const int r = lane + 32 * j;
      pk[j] = r < nrows ? __ldg(kl + r) : 0;
    }
  };
  int staged_seq = -1, staged_layer = -1;
  // element offset of a slot of the current sequence, -1 outside the view
  auto slot_offset = [&](int layer, int seq, int slot) -> int64_t {
    if (!bt_in_smem) return kv_row_offset(kv, layer, seq, slot, dm.T);
    if (slot < 0) return -1;
    const int bi = slot / kv.block_size;
    if (bi >= kv.max_blocks) return -1;
    const int blk = bt_s[bi];
    if (blk < 0 || blk >= kv.num_blocks) return -1;
    return (int64_t)layer * kv.stride_layer + (int64_t)blk * kv.stride_block +
           (int64_t)(slot - bi * kv.block_size) * kv.stride_token;
  };

  // issue the loads of the batch at cursor c (kept slots pk) into stage s
  auto issue = [&](const Cursor& c, const int (&pk)[kMaxRowsPerLane], int s) {
    // the stream's block table (per layer when the layers have their own tables)
    if (bt_in_smem && (c.seq != staged_seq || (kv.table_stride_layer && c.layer != staged_layer))) {
      __syncwarp();
      const int32_t* tab = kv.block_table + (int64_t)c.layer * kv.table_stride_layer + (int64_t)c.seq * kv.max_blocks;
      for (int j = lane; j < kv.max_blocks; j += 32) bt_s[j] = __ldg(tab + j);
      __syncwarp();
      staged_seq = c.seq;
      staged_layer = c.layer;
    }
    const int nrows = min(rpb, c.end - c.i);
    char* kvb = c.kvk ? kv.base[1] : kv.base[0];
    unsigned char* stage = smem + s * kStageBytes;
    const char* src[kMaxRowsPerLane];
    uint32_t total = 0;
#pragma unroll
    for (int j = 0; j < kMaxRowsPerLane; ++j) {
      const int r = lane + 32 * j;
      src[j] = nullptr;
      bool ok = false;
      if (r < nrows) {
        const int i = c.i + r;
        const int from = pk[j];
        const int64_t dof = slot_offset(c.layer, c.seq, i);
        const char* from_ptr = nullptr;
        if (from >= c.stash_at && from < c.n_new) {  // saved before the copy: a later chunk overwrites it
          const int k = i - c.row0;
          if (k >= 0 && k < dm.stash_rows)
            from_ptr = st.stash + ((size_t)(blockIdx.x + 1) * dm.stash_rows + k) * rb;
        } else if (from >= i) {
          const int64_t so = slot_offset(c.layer, c.seq, from);
          if (so >= 0) from_ptr = kvb + (so + c.hg * piece_elems) * 2;
        }
        ok = from_ptr != nullptr && dof >= 0;
        if (ok) {
          src[j] = from_ptr;
          dptr[s][r] = kvb + (dof + c.hg * piece_elems) * 2;
        } else {
          dptr[s][r] = nullptr;
          set_error(st.err, from < i ? EPIKV_DEV_KEPT : EPIKV_DEV_SLOT);
        }
      }
      total += __popc(__ballot_sync(0xffffffffu, ok)) * (uint32_t)rb;
    }
    if (lane == 0) {
      stage_rows[s] = nrows;
      mbar_arrive_expect_tx(&full[s], total);
    }
    __syncwarp();
#pragma unroll
    for (int j = 0; j < kMaxRowsPerLane; ++j)
      if (src[j]) tma_load_1d(stage + (lane + 32 * j) * rb, src[j], rb, &full[s]);
  };

  Cursor ld;
  if (balanced) {
    ld.u = o_begin < o_stop ? 0 : units;
    if (ld.u == 0) open_at(ld, o_begin);
  } else {
    ld.u = kLayers ? next_unit(0) : (int)blockIdx.x;
    load_unit(ld);
  }
  int pk[kMaxRowsPerLane];
  prefetch(ld, pk);
  int k_issue = 0, k_store = 0;
  bool timed_out = false;
  for (int p = 0; p < kStages - 1 && ld.u < units; ++p) {
    issue(ld, pk, k_issue % kStages);
    ++k_issue;
    advance(ld);
    prefetch(ld, pk);
  }
  while (k_store < k_issue) {
    const int s = k_store % kStages;
    if (!mbar_wait_bounded(&full[s], (k_store / kStages) & 1, kWaitNs)) {
      timed_out = true;
      break;
    }
    __syncwarp();
    const int nrows = stage_rows[s];
    unsigned char* stage = smem + s * kStageBytes;
    for (int r = lane; r < nrows; r += 32)
      if (dptr[s][r]) tma_store_1d(dptr[s][r], stage + r * rb, rb);
    tma_commit();
    ++k_store;
    if (ld.u < units) {
      tma_wait_read<1>();  // the stage about to be refilled has been read out
      __syncwarp();
      issue(ld, pk, k_issue % kStages);
      ++k_issue;
      advance(ld);
      prefetch(ld, pk);    // its latency hides behind the next barrier wait
    }
  }
  if (timed_out) {
    if (lane == 0) set_error(st.err, EPIKV_DEV_TIMEOUT);
    // let the loads still in flight land before the CTA's shared memory goes away
    for (int k = k_store; k < k_issue; ++k)
      mbar_wait_bounded(&full[k % kStages], (k / kStages) & 1, kDrainNs);
  }
  tma_wait_all();
  if (kLayers && lane == 0) {
    // every CTA has fetched its last unit once all have counted in: the last resets
    __threadfence();
    if (atomicAdd(st.work + 1, 1u) == gridDim.x - 1) {
      st.work[0] = 0u;
      st.work[1] = 0u;
    }
  }
}

// Before a balanced compaction: where chunk g begins inside a stream (row a),
// CTA g saves into stash g the sources of the previous chunk's rows there
// that lie in [a, n_new) -- the region later chunks overwrite -- row by row
// from the first such row (stash_row0[g]).  Nothing of the cache is written,
// so every read sees the rows as the selection left them.
__global__ void __launch_bounds__(kStashThreads) compact_stash_kernel(DevState st, Dims dm, KvDev kv,
                                                                      const int32_t* __restrict__ seq_ids,
                                                                      int n_seq, const int32_t* __restrict__ kept,
                                                                      int kept_stride) {
  pdl_wait();
  pdl_trigger();
  extern __shared__ __align__(128) unsigned char smem[];
  int* list = reinterpret_cast<int*>(smem);
  int64_t* pre = reinterpret_cast<int64_t*>(list + list_ints(n_seq));
  const bool layers = dm.layer_budgets;
  const int sp = layers ? 2 : 2 * dm.L;  // streams per pair
  __shared__ int s_pairs, s_bal;
  __shared__ int64_t s_rows;
  if (threadIdx.x < 32) {
    const int n_ev = evicting_entries(st, dm, seq_ids, n_seq, list, layers ? nullptr : pre, threadIdx.x);
    const int n_pairs = layers ? n_ev * dm.L : n_ev;
    int64_t rows = 0;
    if (!layers) rows = pre[n_ev];
    else if (n_pairs <= kMaxLayerPairs) rows = layer_pairs(st, dm, seq_ids, list, n_ev, pre, threadIdx.x);
    const bool bal = n_ev > 0 && (!layers || n_pairs <= kMaxLayerPairs) &&
                     balanced_split(st, dm, seq_ids, list, n_ev, kept, kept_stride, layers, n_pairs, rows * sp,
                                    threadIdx.x);
    if (threadIdx.x == 0) {
      s_pairs = n_pairs;
      s_rows = rows;
      s_bal = bal;
    }
  }
  __syncthreads();
  if (!s_bal || blockIdx.x == 0) return;
  const int n_pairs = s_pairs;
  const int64_t total = s_rows * sp;
  const int64_t o = (int64_t)blockIdx.x * total / gridDim.x;
  if (o >= total) return;
  int p, q;
  int64_t r;
  locate_row(pre, n_pairs, sp, o, p, q, r);
  if (r == 0) return;  // the chunk begins its stream: no other chunk reads its region
  const PairAt pa = pair_at(st, dm, seq_ids, list, kept, kept_stride, layers, p, q);
  const int seq = pa.seq, fe = pa.first, n_new = pa.n_new;
  const int a = fe + (int)r;
  const int32_t* kl = pa.kl;
  // the previous chunk's rows in this stream start at seg_start; those whose
  // sources lie in [a, n_new) are a suffix [i0, i1) of them, at most
  // stash_rows long (balanced_split), so inside [lo, a)
  const int64_t s0 = pre[p] * sp + (int64_t)q * (pre[p + 1] - pre[p]);
  const int64_t o_prev = (int64_t)(blockIdx.x - 1) * total / gridDim.x;
  const int seg_start = fe + (int)(o_prev > s0 ? o_prev - s0 : 0);
  const int lo = max(seg_start, a - dm.stash_rows);
  const int t = threadIdx.x;
  __shared__ int s_src[kStashRows];  // the sources of rows lo .. a-1
  const int src = t < a - lo ? __ldg(kl + lo + t) : INT_MAX;
  if (t < a - lo) s_src[t] = src;
  const int i0 = lo + __syncthreads_count(src < a);      // kept is increasing: counts of prefixes
  const int i1 = lo + __syncthreads_count(src < n_new);
  if (t == 0) st.stash_row0[blockIdx.x] = i0;
  const int x = i1 - i0;
  const int layer = pa.layer;
  const char* kvb = pa.kvk ? kv.base[1] : kv.base[0];
  const int v16 = dm.H * dm.d / 8;  // 16-byte vectors per row
  uint4* dst = reinterpret_cast<uint4*>(st.stash + (size_t)blockIdx.x * dm.stash_rows * dm.H * dm.d * 2);
  // each warp copies two rows at a time, every lane's loads issued before its stores
  constexpr int kWarps = kStashThreads / 32;
  const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
  for (int r0 = warp; r0 < x; r0 += 2 * kWarps) {
    const int r1 = r0 + kWarps;
    const int64_t f0 = kv_row_offset(kv, layer, seq, s_src[i0 - lo + r0], dm.T);
    const int64_t f1 = r1 < x ? kv_row_offset(kv, layer, seq, s_src[i0 - lo + r1], dm.T) : -2;
    if ((f0 == -1 || f1 == -1) && lane == 0) set_error(st.err, EPIKV_DEV_SLOT);
    const uint4* p0 = reinterpret_cast<const uint4*>(kvb + f0 * 2);
    const uint4* p1 = reinterpret_cast<const uint4*>(kvb + f1 * 2);
    for (int k0 = lane; k0 < v16; k0 += kStashUnroll * 32) {
      uint4 v0[kStashUnroll], v1[kStashUnroll];
#pragma unroll
      for (int u = 0; u < kStashUnroll; ++u) {
        const int k = k0 + 32 * u;
        if (k < v16) {
          if (f0 >= 0) v0[u] = __ldg(p0 + k);
          if (f1 >= 0) v1[u] = __ldg(p1 + k);
        }
      }
#pragma unroll
      for (int u = 0; u < kStashUnroll; ++u) {
        const int k = k0 + 32 * u;
        if (k < v16) {
          if (f0 >= 0) dst[(size_t)r0 * v16 + k] = v0[u];
          if (f1 >= 0) dst[(size_t)r1 * v16 + k] = v1[u];
        }
      }
    }
  }
}

// The batch entries' evictions have been applied: nothing is left pending.
__global__ void compact_consumed_kernel(DevState st, Dims dm, const int32_t* __restrict__ seq_ids, int n_seq) {
  pdl_wait();
  pdl_trigger();
  for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < n_seq; b += gridDim.x * blockDim.x) {
    const int seq = seq_ids[b];
    if (seq < 0 || seq >= dm.S) continue;
    st.first_changed[seq] = st.n_cache[seq];
    if (dm.layer_budgets)
      for (int l = 0; l < dm.L; ++l) st.lfirst[seq * dm.L + l] = st.n_layer[seq * dm.L + l];
  }
}

static int g_ctas_per_sm = 0;

static size_t stash_smem(int n_seq, int L, bool layers) {
  return (size_t)list_ints(n_seq) * sizeof(int) + (size_t)pre_entries(pairs_cap(n_seq, L, layers)) * sizeof(int64_t);
}

static size_t compact_smem(int n_seq, int L, bool layers) {
  return (size_t)kStages * kStageBytes + stash_smem(n_seq, L, layers) + (size_t)kStagedBlocks * sizeof(int);
}

cudaError_t compact_prepare(int device, int* ctas_per_sm) {
  (void)device;
  const int mx = (int)compact_smem(4096, 64, true);  // the largest batch and pair table
  cudaError_t e = cudaSuccess;
  auto allow = [&](auto kern) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  };
  allow(compact_kernel<false, true>);
  allow(compact_kernel<true, true>);
  allow(compact_kernel<true, false>);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(compact_stash_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)stash_smem(4096, 64, true));
  if (e != cudaSuccess) return e;
  int n = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, compact_kernel<false, true>, 32, compact_smem(64, 32, false));
  if (e != cudaSuccess) return e;
  g_ctas_per_sm = n > 0 ? n : 1;
  if (EPIKV_COMPACT_CTAS_PER_SM > 0 && EPIKV_COMPACT_CTAS_PER_SM < g_ctas_per_sm)
    g_ctas_per_sm = EPIKV_COMPACT_CTAS_PER_SM;
  if (ctas_per_sm) *ctas_per_sm = g_ctas_per_sm;
  return cudaSuccess;
}

cudaError_t launch_compact(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                           const int32_t* kept, int kept_stride, const KvDev& kv, int ctas,
                           cudaStream_t stream, int* launches) {
  if (n_seq == 0) return cudaSuccess;
  const bool layers = dm.layer_budgets;
  const bool split = !layers || n_seq * dm.L <= kMaxLayerPairs;  // the balanced split may apply
  const size_t smem = compact_smem(n_seq, dm.L, layers);
  if (split && ctas <= kMaxStashCtas) {  // the balanced split's stash (the kernel checks whether it applies)
    pdl_launch(compact_stash_kernel, ctas, kStashThreads, stash_smem(n_seq, dm.L, layers), stream, st, dm, kv,
               seq_ids, n_seq, kept, kept_stride);
    ++*launches;
    const cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  auto go = [&](auto kern) {
    plain_launch(kern, ctas, 32, smem, stream, st, dm, kv, seq_ids, n_seq, kept, kept_stride);
  };
  if (!layers) go(compact_kernel<false, true>);
  else if (split) go(compact_kernel<true, true>);
  else go(compact_kernel<true, false>);
  ++*launches;
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  pdl_launch(compact_consumed_kernel, (n_seq + 255) / 256, 256, 0, stream, st, dm, seq_ids, n_seq);
  ++*launches;
  return cudaGetLastError();
}

}  // namespace epikv
