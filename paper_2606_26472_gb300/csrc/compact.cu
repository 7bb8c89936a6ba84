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
// In-place safety without any inter-CTA wait: streams are disjoint bytes, so
// one CTA owns each; inside a stream kept[i] >= i and rows are processed in
// increasing i, so a load (slot kept[i] >= i) never reads a slot that an
// earlier store has written, and a later store to a slot some earlier batch
// still had to read is issued only after that batch's loads completed.
//
// Under per-layer budgets (kLayers) each (sequence, layer) has its own kept
// list, first moved slot and length; the streams and the copy are unchanged.
// The streams then differ in length (a layer's rows follow its budget), so
// the CTAs take units from a shared counter instead of a fixed stride, in
// layer-major order: with budgets that fall with depth, larger streams come
// first and the greedy assignment ends nearly level.
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

#ifndef EPIKV_COMPACT_STAGED_BLOCKS
#define EPIKV_COMPACT_STAGED_BLOCKS 1024  // block-table entries kept in shared memory (larger tables: global reads)
#endif
constexpr int kStagedBlocks = EPIKV_COMPACT_STAGED_BLOCKS;

struct Cursor {
  int u;      // unit index (this CTA strides by gridDim.x)
  int i;      // next row of the unit
  int end;    // row past the last of the unit
  int b, seq, layer, kvk, hg;
};

template <bool kLayers>
__global__ void __launch_bounds__(32) compact_kernel(DevState st, Dims dm, KvDev kv,
                                                     const int32_t* __restrict__ seq_ids, int n_seq,
                                                     const int32_t* __restrict__ kept, int kept_stride) {
  extern __shared__ __align__(128) unsigned char smem[];
  __shared__ __align__(8) uint64_t full[kStages];
  __shared__ char* dptr[kStages][kMaxRPB];
  __shared__ int stage_rows[kStages];
  int* list = reinterpret_cast<int*>(smem + kStages * kStageBytes);
  int* bt_s = list + (n_seq + 31) / 32 * 32;  // the current sequence's block table
  const int lane = threadIdx.x;

  // ---- the batch entries that evicted (every CTA builds the same list)
  int n_ev = 0;
  for (int base = 0; base < n_seq; base += 32) {
    const int b = base + lane;
    bool ev = false;
    if (b < n_seq) {
      const int seq = seq_ids[b];
      ev = seq >= 0 && seq < dm.S && st.first_changed[seq] < st.n_cache[seq];
    }
    const unsigned m = __ballot_sync(0xffffffffu, ev);
    if (ev) list[n_ev + __popc(m & ((1u << lane) - 1u))] = b;
    n_ev += __popc(m);
  }
  __syncwarp();
  if (n_ev == 0) return;

  // ---- head split: whole token rows unless too few streams evict to give
  // every CTA one (small TMA copies cost much more per byte than a tail)
  const int G = gridDim.x;
  int hs = 1;
#if EPIKV_COMPACT_HEAD_SPLIT > 0
  if (dm.H % EPIKV_COMPACT_HEAD_SPLIT == 0) hs = EPIKV_COMPACT_HEAD_SPLIT;
#else
  while ((long)n_ev * 2 * dm.L * hs < G && dm.H % (2 * hs) == 0 && (dm.H / (2 * hs)) * dm.d * 2 >= 256) hs *= 2;
#endif
  const int rb = (dm.H / hs) * dm.d * 2;               // bytes per row piece
  const int64_t piece_elems = (int64_t)(dm.H / hs) * dm.d;
  const int rpb = min(kStageBytes / rb, kMaxRPB);      // rows per batch
  const int upe = 2 * dm.L * hs;
  const int units = n_ev * upe;
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
      if (c.i < c.end) return;
      c.u = next_unit(c.u);
    }
  };
  auto advance = [&](Cursor& c) {
    c.i += rpb;
    if (c.i >= c.end) {
      c.u = next_unit(c.u);
      load_unit(c);
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
        const int64_t so = from >= i ? slot_offset(c.layer, c.seq, from) : -1;
        const int64_t dof = slot_offset(c.layer, c.seq, i);
        ok = so >= 0 && dof >= 0;
        if (ok) {
          src[j] = kvb + (so + c.hg * piece_elems) * 2;
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
  ld.u = kLayers ? next_unit(0) : (int)blockIdx.x;
  load_unit(ld);
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

// The batch entries' evictions have been applied: nothing is left pending.
__global__ void compact_consumed_kernel(DevState st, Dims dm, const int32_t* __restrict__ seq_ids, int n_seq) {
  for (int b = blockIdx.x * blockDim.x + threadIdx.x; b < n_seq; b += gridDim.x * blockDim.x) {
    const int seq = seq_ids[b];
    if (seq < 0 || seq >= dm.S) continue;
    st.first_changed[seq] = st.n_cache[seq];
    if (dm.layer_budgets)
      for (int l = 0; l < dm.L; ++l) st.lfirst[seq * dm.L + l] = st.n_layer[seq * dm.L + l];
  }
}

static int g_ctas_per_sm = 0;

static size_t compact_smem(int n_seq) {
  return (size_t)kStages * kStageBytes + (size_t)((n_seq + 31) / 32 * 32) * sizeof(int) +
         (size_t)kStagedBlocks * sizeof(int);
}

cudaError_t compact_prepare(int device, int* ctas_per_sm) {
  (void)device;
  cudaError_t e = cudaFuncSetAttribute(compact_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)compact_smem(4096));
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(compact_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)compact_smem(4096));
  if (e != cudaSuccess) return e;
  int n = 0;
  e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, compact_kernel<false>, 32, compact_smem(64));
  if (e != cudaSuccess) return e;
  g_ctas_per_sm = n > 0 ? n : 1;
  if (EPIKV_COMPACT_CTAS_PER_SM > 0 && EPIKV_COMPACT_CTAS_PER_SM < g_ctas_per_sm) g_ctas_per_sm = EPIKV_COMPACT_CTAS_PER_SM;
  if (ctas_per_sm) *ctas_per_sm = g_ctas_per_sm;
  return cudaSuccess;
}

cudaError_t launch_compact(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                           const int32_t* kept, int kept_stride, const KvDev& kv, int ctas,
                           cudaStream_t stream, int* launches) {
  if (n_seq == 0) return cudaSuccess;
  if (dm.layer_budgets)
    compact_kernel<true><<<ctas, 32, compact_smem(n_seq), stream>>>(st, dm, kv, seq_ids, n_seq, kept, kept_stride);
  else
    compact_kernel<false><<<ctas, 32, compact_smem(n_seq), stream>>>(st, dm, kv, seq_ids, n_seq, kept, kept_stride);
  ++*launches;
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  compact_consumed_kernel<<<(n_seq + 255) / 256, 256, 0, stream>>>(st, dm, seq_ids, n_seq);
  ++*launches;
  return cudaGetLastError();
}

}  // namespace epikv
