// Top-K retention under the budget (Sec. 3.1, Sec. 3.3, App. D).
//
// One 1024-thread CTA per sequence.  Prefill slots and the trailing recency
// window R = min(cap, K/4) are always kept; the remaining M = K - P - R slots
// go to the highest-scoring candidates.  The M-th largest score is found
// exactly by a 4-pass 8-bit radix select over order-preserving u32 keys
// (NaN lowest, -0 == +0); candidates above the threshold are kept, and of the
// candidates equal to it the lowest slots are kept.  Two block-wide ordered
// scans emit the kept list in ascending slot order.  The slot metadata
// (scores of every kind and positions) is then compacted in place, which is
// safe in increasing order because kept[i] >= i.  When the cache has at most
// kSelStagedMax slots the candidates' keys are first staged in shared memory,
// and the radix passes and scans read them there; when the metadata columns
// (at most kFusedCols) and the kept list fit beside them, the columns are
// staged in the same loads, so the moved rows are written from shared memory
// (coalesced) as soon as the kept list is known.
//
// Chunk-level selection (select_chunk = C > 1; the paper names chunk-level
// scoring as future work, Sec. 5): a first pass gives every candidate slot the
// key of its position chunk floor(pos / C), the fp32 mean of the chunk's
// candidate scores summed in slot order by the thread that owns the chunk's
// first slot.  Chunks are runs of consecutive slots (positions increase with
// the slot), so the unchanged selection on those keys -- larger keys first,
// equal keys lowest slot first -- keeps whole chunks in rank order, ties to
// the earlier chunk, and the lowest slots of the first chunk that does not
// fit.
//
// Per-layer budgets (layer_budgets; the paper names per-layer budgets as
// future work, Sec. 5): every layer evicts its own cache with its own budget
// K_l, all layers keep the prefill and one recency window R (from the
// smallest budget) and evict at the same events.  Under those rules a layer's
// cache is always its own budget's selection from any larger layer's cache,
// so one ranking serves every layer: the context keeps the largest layer's
// slots (the union of all layers) with a 64-bit mask per slot of the layers
// holding it.  layer_keep_kernel (a CTA per layer and sequence) finds layer
// l's threshold of M_l = K_l - P - R over the union's candidates, writes the
// layer's kept list in its own slot numbering and a keep bit per union slot
// (a 32-bit word per 32 slots); layer_union_kernel (a CTA per sequence) turns
// the keep bits into the new masks and compacts the union's metadata.
#include <cooperative_groups.h>

#include "common.cuh"
#include "kernels.h"

namespace epikv {

#ifndef EPIKV_SEL_CLUSTER_MIN
// token budgets: caches of more slots than this take the cluster kernel, the
// others one CTA per sequence (measured per evicting sequence, one CTA /
// cluster of 8: 8,320 slots 26 / 54 us, a one-token ragged eviction 21 /
// 39 us, 2,048 slots 14 / 32 us; 4 x 65,536 slots 218 / 70 us)
#define EPIKV_SEL_CLUSTER_MIN 24576
#endif
#ifndef EPIKV_SEL_THREADS
// threads of the selection CTA (measured per evicting sequence, 1024 / 512 /
// 256: one-token decode of 64 sequences 20.7 / 23.9 / 30.7 us; 8,320 slots
// 26.1 / 29.6 / 43.1 us; 65,536 slots 223 / 300 / 471 us)
#define EPIKV_SEL_THREADS 1024
#endif
constexpr int kSelThreads = EPIKV_SEL_THREADS;

__device__ __forceinline__ uint32_t order_key(float f) {
  if (f != f) return 0u;          // NaN below every number
  if (f == 0.0f) f = 0.0f;        // -0 == +0
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive prefix sum over the block of NT threads; *total receives the sum.
template <int NT = kSelThreads>
__device__ __forceinline__ int block_exclusive_scan(int v, int* total, int* sh /*[32]*/) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) sh[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < (NT / 32) ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;  // inclusive warp totals
  }
  __syncthreads();
  const int before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[NT / 32 - 1];
  __syncthreads();
  return before;
}

template <int NT = kSelThreads>
__device__ __forceinline__ int block_min(int v, int* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int w = lane < (NT / 32) ? sh[lane] : INT_MAX;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w = min(w, __shfl_xor_sync(0xffffffffu, w, o));
    if (lane == 0) sh[0] = w;
  }
  __syncthreads();
  const int r = sh[0];
  __syncthreads();
  return r;
}

// Slot j <- slot kept[j] of the sequence's scores (every kind) and positions,
// for j from fe to n_kept, in place: safe in increasing j because kept[j] >= j
// and each round reads all its sources before any of its stores.  A round
// stages as many rows as `stage` (stage_words 32-bit words of shared memory,
// free by now) holds, all their loads in flight together; without room for
// a round of kSelThreads rows, a round is one row per thread in registers.
// Every thread of the block calls it.
__device__ __forceinline__ void compact_metadata(const DevState& st, const Dims& dm, int seq,
                                                 const int32_t* __restrict__ kept, int fe, int n_kept,
                                                 uint32_t* stage, int stage_words) {
  const int tid = threadIdx.x;
  int32_t* ps = st.pos + (size_t)seq * dm.T;
  const size_t base = (size_t)seq * dm.T;
  unsigned on = 0;  // the score kinds held
#pragma unroll
  for (int k = 0; k < kNumKinds; ++k) on |= (st.score[k] != nullptr ? 1u : 0u) << k;
  const int n_on = __popc(on);
  const int cap = stage_words / (n_on + 1);
  if (cap >= kSelThreads) {
    constexpr int U = 4;  // rows per thread with their loads in flight together
    for (int j0 = fe; j0 < n_kept; j0 += cap) {
      const int m = min(cap, n_kept - j0);
      for (int r0 = tid; r0 < m; r0 += U * kSelThreads) {
        int src[U];
#pragma unroll
        for (int u = 0; u < U; ++u) src[u] = r0 + u * kSelThreads < m ? kept[j0 + r0 + u * kSelThreads] : -1;
        uint32_t v[U][kNumKinds + 1];
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (src[u] < 0) continue;
#pragma unroll
          for (int k = 0; k < kNumKinds; ++k)
            if (on >> k & 1u) v[u][k] = __float_as_uint(st.score[k][base + src[u]]);
          v[u][kNumKinds] = (uint32_t)ps[src[u]];
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
          if (src[u] < 0) continue;
          const int r = r0 + u * kSelThreads;
#pragma unroll
          for (int k = 0; k < kNumKinds; ++k)
            if (on >> k & 1u) stage[__popc(on & ((1u << k) - 1u)) * cap + r] = v[u][k];
          stage[n_on * cap + r] = v[u][kNumKinds];
        }
      }
      __syncthreads();
      for (int r = tid; r < m; r += kSelThreads) {
        int q = 0;
#pragma unroll
        for (int k = 0; k < kNumKinds; ++k)
          if (st.score[k]) st.score[k][base + j0 + r] = __uint_as_float(stage[(q++) * cap + r]);
        ps[j0 + r] = (int32_t)stage[n_on * cap + r];
      }
      __syncthreads();
    }
    return;
  }
  for (int j0 = fe; j0 < n_kept; j0 += kSelThreads) {
    const int j = j0 + tid;
    float v[kNumKinds];
    int32_t p = 0;
    if (j < n_kept) {
      const int src = kept[j];
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k) v[k] = st.score[k] ? st.score[k][(size_t)seq * dm.T + src] : 0.f;
      p = ps[src];
    }
    __syncthreads();
    if (j < n_kept) {
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k)
        if (st.score[k]) st.score[k][(size_t)seq * dm.T + j] = v[k];
      ps[j] = p;
    }
    __syncthreads();
  }
}

// Metadata columns (score kinds + positions) the selection stages beside its
// keys; contexts with more score kinds move their metadata after selecting.
constexpr int kFusedCols = 3;
#ifndef EPIKV_SEL_FUSED_META
#define EPIKV_SEL_FUSED_META 1  // 0: the metadata always moved after selecting (compact_metadata)
#endif

struct RadixShared {
  uint32_t hist[256];
  uint32_t prefix, mask, remaining;
};

// The M-th largest key_at(i) over i in [c0, c1), 0 < M <= c1 - c0, by a
// 4-pass 8-bit radix select: *theta is that key, *need_eq the number of
// keys equal to it that belong to the M largest (the lowest slots first) and
// *total_eq (when given) the number of keys equal to it.
// Every thread of the block (NT threads) calls it.
template <int NT = kSelThreads, typename KeyAt>
__device__ __forceinline__ void radix_select(const KeyAt& key_at, int c0, int c1, int M, RadixShared& rs,
                                             uint32_t* theta, int* need_eq, int* total_eq = nullptr) {
  const int tid = threadIdx.x;
  __syncthreads();  // every thread has read the previous call's result
  if (tid == 0) {
    rs.prefix = 0u;
    rs.mask = 0u;
    rs.remaining = (uint32_t)M;
  }
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int j = tid; j < 256; j += NT) rs.hist[j] = 0u;
    __syncthreads();
    const uint32_t prefix = rs.prefix, mask = rs.mask;
    for (int i = c0 + tid; i < c1; i += NT) {
      const uint32_t k = key_at(i);
      if ((k & mask) == prefix) atomicAdd(&rs.hist[(k >> shift) & 255u], 1u);
    }
    __syncthreads();
    if (tid < 32) {
      // lane l owns digits 255-8l .. 248-8l (descending)
      const int lane = tid;
      uint32_t lsum = 0;
#pragma unroll
      for (int j = 0; j < 8; ++j) lsum += rs.hist[255 - 8 * lane - j];
      uint32_t incl = lsum;
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
      }
      const uint32_t rem = rs.remaining;
      const unsigned hit = __ballot_sync(0xffffffffu, incl >= rem);
      const int owner = __ffs(hit) - 1;  // first lane reaching the target
      if (lane == owner) {
        uint32_t before = incl - lsum;
        for (int j = 0; j < 8; ++j) {
          const int dg = 255 - 8 * lane - j;
          if (before + rs.hist[dg] >= rem) {
            rs.prefix = prefix | ((uint32_t)dg << shift);
            rs.mask = mask | (255u << shift);
            rs.remaining = rem - before;
            break;
          }
          before += rs.hist[dg];
        }
      }
    }
    __syncthreads();
  }
  *theta = rs.prefix;
  *need_eq = (int)rs.remaining;
  if (total_eq) *total_eq = (int)rs.hist[rs.prefix & 255u];  // the last pass's bin: keys equal to theta
}

template <bool kChunked>
__global__ void __launch_bounds__(kSelThreads) select_kernel(DevState st, Dims dm,
                                                             const int32_t* __restrict__ seq_ids,
                                                             const int32_t* __restrict__ budget,
                                                             const int32_t* __restrict__ trigger,
                                                             int32_t* __restrict__ kept_out, int kept_stride,
                                                             int32_t* __restrict__ n_kept_out, int staged_cap,
                                                             int smem_words) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.x, tid = threadIdx.x;
  const int seq = seq_ids[b];
  if (seq < 0 || seq >= dm.S) {
    if (tid == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  const int n = st.n_cache[seq];
  const int K = budget[b];
  if (K < 1 || K > dm.T) {
    if (tid == 0) {
      set_error(st.err, EPIKV_DEV_BUDGET);
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const int trig = trigger ? trigger[b] : K;
  if (n <= K || n <= trig) {  // nothing to evict
    if (tid == 0) {
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const int P = min(st.prefill[seq], n);
  const int R = min(min(dm.recency_cap, K / 4), max(0, K - P));
  const int M = max(0, K - P - R);
  const int c0 = P, c1 = n - R;  // candidates [c0, c1)
  if (max(K, P) > kept_stride) {
    if (tid == 0) {
      set_error(st.err, EPIKV_DEV_KEPT);
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const float* __restrict__ sc = st.score[kind_index(st.policy[seq])] + (size_t)seq * dm.T;
  int32_t* out = kept_out + (size_t)b * kept_stride;

  // ---- chunk keys (chunk-level selection only)
  uint32_t* __restrict__ ck = kChunked ? st.ckey + (size_t)seq * dm.T : nullptr;
  if (kChunked) {
    const int C = dm.select_chunk;
    const int32_t* __restrict__ pz = st.pos + (size_t)seq * dm.T;
    for (int i = c0 + tid; i < c1; i += kSelThreads) {
      const int c = pz[i] / C;
      if (i > c0 && pz[i - 1] / C == c) continue;  // not the chunk's first candidate
      float s = 0.f;
      int j = i;
      for (; j < c1 && pz[j] / C == c; ++j) s = __fadd_rn(s, sc[j]);  // at most C members
      const uint32_t k = order_key(__fdiv_rn(s, (float)(j - i)));
      for (int q = i; q < j; ++q) ck[q] = k;
    }
    __syncthreads();
  }
  // the candidates' keys staged in shared memory when the launch provided room
  // for the cache (every later pass reads them there instead of from L2)
  extern __shared__ uint32_t skey[];
  const bool staged = staged_cap >= c1 - c0;
  // With at most kFusedCols metadata columns (each kind's scores, then the
  // positions) and room for all of them, the cache's columns are staged too,
  // from the first candidate on (no slot before it moves): the kept rows are
  // then written from shared memory as the kept list is emitted, with no
  // round trip after the selection.
  __shared__ uint32_t* s_col[kNumKinds + 1];
  __shared__ int s_ncol;
  if (tid == 0) {
    int q = 0;
    for (int k = 0; k < kNumKinds; ++k)
      if (st.score[k]) s_col[q++] = reinterpret_cast<uint32_t*>(st.score[k]) + (size_t)seq * dm.T;
    s_col[q++] = reinterpret_cast<uint32_t*>(st.pos) + (size_t)seq * dm.T;
    s_ncol = q;
  }
  __syncthreads();
  const int ncol = s_ncol;
  const int kpad = (c1 - c0 + 3) & ~3;
  const bool fused = EPIKV_SEL_FUSED_META && staged && ncol <= kFusedCols &&
                     (int64_t)kpad + (int64_t)(ncol + 1) * n <= smem_words;
  uint32_t* smeta = skey + kpad;  // fused: [ncol][n], column c of slot i at c * n + i
  int* skept = reinterpret_cast<int*>(smeta + (size_t)ncol * n);  // fused: the kept list
  uint32_t* col[kFusedCols];
#pragma unroll
  for (int c = 0; c < kFusedCols; ++c) col[c] = c < ncol ? s_col[c] : nullptr;
  if (staged) {
    // U slots per thread with every load in flight before the stores
    constexpr int U = 4;
    const int hi = fused ? n : c1;
    for (int i0 = c0 + tid; i0 < hi; i0 += U * kSelThreads) {
      uint32_t kv[U], mv[U][kFusedCols];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int i = i0 + u * kSelThreads;
        if (i < c1) kv[u] = kChunked ? ck[i] : order_key(sc[i]);
#pragma unroll
        for (int c = 0; c < kFusedCols; ++c)
          if (fused && c < ncol && i < n) mv[u][c] = __ldcg(col[c] + i);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int i = i0 + u * kSelThreads;
        if (i < c1) skey[i - c0] = kv[u];
#pragma unroll
        for (int c = 0; c < kFusedCols; ++c)
          if (fused && c < ncol && i < n) smeta[c * n + i] = mv[u][c];
      }
    }
    __syncthreads();
  }
  auto key_at = [&](int i) -> uint32_t {
    if (staged) return skey[i - c0];
    return kChunked ? ck[i] : order_key(sc[i]);
  };

  __shared__ RadixShared rs;
  __shared__ int sh_scan[32];

  // ---- radix select of the M-th largest key among the candidates
  uint32_t theta = 0xFFFFFFFFu;
  int need_eq = 0, total_eq = 0;  // no key is 0xFFFFFFFF (order_key), so M == 0 keeps no candidate
  if (M > 0) radix_select(key_at, c0, c1, M, rs, &theta, &need_eq, &total_eq);

  // ---- ordered scans over contiguous per-thread slot ranges
  const int per = (n + kSelThreads - 1) / kSelThreads;
  const int a = min(n, tid * per), e = min(n, a + per);
  // when every key equal to theta is kept (the usual case), which of them
  // come first does not matter and the count before each thread is not needed
  const bool all_eq = need_eq == total_eq;
  int eq_base = 0;
  if (!all_eq) {  // uniform across the block
    int eq_local = 0;
    for (int i = max(a, c0); i < min(e, c1); ++i) eq_local += (key_at(i) == theta);
    int tot;
    eq_base = block_exclusive_scan(eq_local, &tot, sh_scan);
  }

  auto kept_slot = [&](int i, int& eqs) -> bool {
    if (i < c0 || i >= c1) return true;
    const uint32_t k = key_at(i);
    return k > theta || (k == theta && (all_eq || eqs++ < need_eq));
  };
  int keep_local = 0, first_ev = INT_MAX;
  uint64_t kmask = 0;  // with at most 64 slots per thread: bit i - a set when slot i is kept
  {
    int eqs = eq_base;
    for (int i = a; i < e; ++i) {
      if (kept_slot(i, eqs)) {
        ++keep_local;
        if (per <= 64) kmask |= 1ull << (i - a);
      } else {
        first_ev = min(first_ev, i);
      }
    }
  }
  int n_kept;
  const int keep_base = block_exclusive_scan(keep_local, &n_kept, sh_scan);
  {
    int o = keep_base;
    if (per <= 64) {  // uniform across the block
      for (uint64_t m = kmask; m; m &= m - 1) {
        const int i = a + __ffsll((long long)m) - 1;
        out[o] = i;
        if (fused) skept[o] = i;
        ++o;
      }
    } else {
      int eqs = eq_base;
      for (int i = a; i < e; ++i)
        if (kept_slot(i, eqs)) out[o++] = i;
    }
  }
  const int fe = min(block_min(first_ev, sh_scan), n_kept);
  __syncthreads();  // kept list visible to the whole block

  // ---- compact slot metadata in place (kept[i] >= i, increasing i); the
  // staged keys are no longer needed, so their shared memory stages it
  // (fused: every row from the staged columns, coalesced stores)
  if (fused) {
    for (int o = fe + tid; o < n_kept; o += kSelThreads) {
      const int i = skept[o];
#pragma unroll
      for (int c = 0; c < kFusedCols; ++c)
        if (c < ncol) col[c][o] = smeta[c * n + i];
    }
  } else {
    compact_metadata(st, dm, seq, out, fe, n_kept, skey, smem_words);
  }
  if (tid == 0) {
    st.n_cache[seq] = n_kept;
    st.first_changed[seq] = fe;
    if (n_kept_out) n_kept_out[b] = n_kept;
    atomicAdd(&st.stats[1], 1ull);
    atomicAdd(&st.stats[2], (unsigned long long)(n_kept - fe));
    atomicAdd(&st.stats[3], (unsigned long long)(n_kept - fe) * (unsigned long long)dm.L);
  }
}

// ---------------------------------------------------------------- token budgets on a thread-block cluster
//
// One sequence's selection spread over a cluster of kCluCtas CTAs (DSMEM for
// the merges, cluster barriers between phases; every CTA of a cluster takes
// the same path, so none leaves while the others wait).  The sequence's slots
// [0, n) are cut into one contiguous slice per CTA.  The radix passes count
// each slice's candidate keys into the CTA's own 256-bin histogram (double
// buffered: a pass's bins are read by the other CTAs until the next pass's
// barrier); after the barrier every CTA reads all kCluCtas histograms and
// takes the same decision.  The ordered scans publish each CTA's counts (keys
// equal to the threshold, kept slots, first evicted slot) for the others'
// prefixes.  The slot metadata is compacted in rounds of destination rows:
// every CTA stages its part of the round's sources, a barrier, then the
// writes (a round's sources lie at or after its destinations' end, so they
// are not written by the round).  Results equal select_kernel's bit for bit.
constexpr int kCluCtas = 8;
constexpr int kCluThreads = 512;
constexpr int kCluStageWords = 8192;   // 32 KiB: a slice's staged keys, then a round's metadata

struct CluShared {
  uint32_t hist[2][256];
  uint32_t prefix, mask, remaining;
  int pub[3];        // this CTA's equal-key count, kept count, first evicted slot
  int sh_scan[32];
};

__global__ void __cluster_dims__(kCluCtas, 1, 1) __launch_bounds__(kCluThreads)
    select_cluster_kernel(DevState st, Dims dm, const int32_t* __restrict__ seq_ids,
                          const int32_t* __restrict__ budget, const int32_t* __restrict__ trigger,
                          int32_t* __restrict__ kept_out, int kept_stride, int32_t* __restrict__ n_kept_out) {
  pdl_wait();
  pdl_trigger();
  namespace cg = cooperative_groups;
  cg::cluster_group cluster = cg::this_cluster();
  constexpr int NT = kCluThreads;
  const int rank = (int)cluster.block_rank();
  const int b = blockIdx.x / kCluCtas, tid = threadIdx.x;
  const bool lead = rank == 0 && tid == 0;
  const int seq = seq_ids[b];
  if (seq < 0 || seq >= dm.S) {
    if (lead) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  const int n = st.n_cache[seq];
  const int K = budget[b];
  if (K < 1 || K > dm.T) {
    if (lead) {
      set_error(st.err, EPIKV_DEV_BUDGET);
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const int trig = trigger ? trigger[b] : K;
  if (n <= K || n <= trig) {  // nothing to evict
    if (lead) {
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const int P = min(st.prefill[seq], n);
  const int R = min(min(dm.recency_cap, K / 4), max(0, K - P));
  const int M = max(0, K - P - R);
  const int c0 = P, c1 = n - R;  // candidates [c0, c1)
  if (max(K, P) > kept_stride) {
    if (lead) {
      set_error(st.err, EPIKV_DEV_KEPT);
      st.first_changed[seq] = n;
      if (n_kept_out) n_kept_out[b] = n;
    }
    return;
  }
  const float* __restrict__ sc = st.score[kind_index(st.policy[seq])] + (size_t)seq * dm.T;
  int32_t* out = kept_out + (size_t)b * kept_stride;
  __shared__ CluShared cs;
  extern __shared__ uint32_t stage[];   // kCluStageWords

  // this CTA's slice of the slots and its candidates
  const int s0 = (int)((int64_t)n * rank / kCluCtas), s1 = (int)((int64_t)n * (rank + 1) / kCluCtas);
  const int a0 = max(s0, c0), a1 = max(a0, min(s1, c1));
  const bool staged = a1 - a0 <= kCluStageWords;
  if (staged) {
    for (int i = a0 + tid; i < a1; i += NT) stage[i - a0] = order_key(sc[i]);
    __syncthreads();
  }
  auto key_at = [&](int i) -> uint32_t { return staged ? stage[i - a0] : order_key(sc[i]); };

  // ---- radix select of the M-th largest candidate key over the cluster
  uint32_t prefix = 0u, mask = 0u, remaining = (uint32_t)M;
  if (M > 0) {
    for (int pass = 0, shift = 24; shift >= 0; ++pass, shift -= 8) {
      uint32_t* h = cs.hist[pass & 1];
      for (int j = tid; j < 256; j += NT) h[j] = 0u;
      __syncthreads();
      for (int i = a0 + tid; i < a1; i += NT) {
        const uint32_t k = key_at(i);
        if ((k & mask) == prefix) atomicAdd(&h[(k >> shift) & 255u], 1u);
      }
      cluster.sync();   // every CTA's bins of this pass are complete
      if (tid < 32) {
        // lane l owns digits 255-8l .. 248-8l (descending), summed over the cluster
        const int lane = tid;
        uint32_t cnt[8], lsum = 0;
#pragma unroll
        for (int j = 0; j < 8; ++j) cnt[j] = 0;
        for (int r = 0; r < kCluCtas; ++r) {
          const uint32_t* hr = cluster.map_shared_rank(h, r);
#pragma unroll
          for (int j = 0; j < 8; ++j) cnt[j] += hr[255 - 8 * lane - j];
        }
#pragma unroll
        for (int j = 0; j < 8; ++j) lsum += cnt[j];
        uint32_t incl = lsum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        const unsigned hit = __ballot_sync(0xffffffffu, incl >= remaining);
        const int owner = __ffs(hit) - 1;  // first lane reaching the target
        if (lane == owner) {
          uint32_t before = incl - lsum;
          for (int j = 0; j < 8; ++j) {
            if (before + cnt[j] >= remaining) {
              cs.prefix = prefix | ((uint32_t)(255 - 8 * lane - j) << shift);
              cs.mask = mask | (255u << shift);
              cs.remaining = remaining - before;
              break;
            }
            before += cnt[j];
          }
        }
      }
      __syncthreads();
      prefix = cs.prefix;
      mask = cs.mask;
      remaining = cs.remaining;
    }
  }
  const uint32_t theta = M > 0 ? prefix : 0xFFFFFFFFu;
  const int need_eq = M > 0 ? (int)remaining : 0;

  // ---- ordered scans: contiguous per-thread ranges of the slice, CTA
  // prefixes from the lower ranks' published counts
  const int per = (s1 - s0 + NT - 1) / NT;
  const int ta = min(s1, s0 + tid * per), te = min(s1, ta + per);
  int eq_local = 0;
  for (int i = max(ta, c0); i < min(te, c1); ++i) eq_local += (key_at(i) == theta);
  int eq_cta;
  int eqs = block_exclusive_scan<NT>(eq_local, &eq_cta, cs.sh_scan);
  if (tid == 0) cs.pub[0] = eq_cta;
  cluster.sync();
  for (int r = 0; r < rank; ++r) eqs += cluster.map_shared_rank(cs.pub, r)[0];
  int keep_local = 0, first_ev = INT_MAX;
  {
    int e = eqs;
    for (int i = ta; i < te; ++i) {
      bool keep = (i < c0) || (i >= c1);
      if (!keep) {
        const uint32_t k = key_at(i);
        keep = k > theta || (k == theta && e++ < need_eq);
      }
      if (keep) ++keep_local; else first_ev = min(first_ev, i);
    }
  }
  int keep_cta;
  int o = block_exclusive_scan<NT>(keep_local, &keep_cta, cs.sh_scan);
  const int fe_cta = block_min<NT>(first_ev, cs.sh_scan);
  if (tid == 0) {
    cs.pub[1] = keep_cta;
    cs.pub[2] = fe_cta;
  }
  cluster.sync();
  int n_kept = 0, fe = INT_MAX;
  for (int r = 0; r < kCluCtas; ++r) {
    const int* pr = cluster.map_shared_rank(cs.pub, r);
    if (r < rank) o += pr[1];
    n_kept += pr[1];
    fe = min(fe, pr[2]);
  }
  fe = min(fe, n_kept);
  {
    int e = eqs;
    for (int i = ta; i < te; ++i) {
      bool keep = (i < c0) || (i >= c1);
      if (!keep) {
        const uint32_t k = key_at(i);
        keep = k > theta || (k == theta && e++ < need_eq);
      }
      if (keep) out[o++] = i;
    }
  }
  cluster.sync();   // the whole kept list is written and visible to the cluster (and no DSMEM read is pending)

  // ---- slot metadata in place, in rounds of destination rows
  int32_t* ps = st.pos + (size_t)seq * dm.T;
  const size_t base = (size_t)seq * dm.T;
  unsigned on = 0;
#pragma unroll
  for (int k = 0; k < kNumKinds; ++k) on |= (st.score[k] != nullptr ? 1u : 0u) << k;
  const int n_on = __popc(on);
  const int rpc = kCluStageWords / (n_on + 1);   // rows of a CTA per round
  for (int j0 = fe; j0 < n_kept; j0 += kCluCtas * rpc) {
    const int r0 = j0 + rank * rpc, r1 = min(n_kept, r0 + rpc);
    for (int j = r0 + tid; j < r1; j += NT) {
      const int src = out[j];
      int q = 0;
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k)
        if (on >> k & 1u) stage[(q++) * rpc + (j - r0)] = __float_as_uint(st.score[k][base + src]);
      stage[n_on * rpc + (j - r0)] = (uint32_t)ps[src];
    }
    cluster.sync();   // every source of the round is read before any of its rows is written
    for (int j = r0 + tid; j < r1; j += NT) {
      int q = 0;
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k)
        if (on >> k & 1u) st.score[k][base + j] = __uint_as_float(stage[(q++) * rpc + (j - r0)]);
      ps[j] = (int32_t)stage[n_on * rpc + (j - r0)];
    }
    __syncthreads();  // the stage is reused by the next round
  }
  if (lead) {
    st.n_cache[seq] = n_kept;
    st.first_changed[seq] = fe;
    if (n_kept_out) n_kept_out[b] = n_kept;
    atomicAdd(&st.stats[1], 1ull);
    atomicAdd(&st.stats[2], (unsigned long long)(n_kept - fe));
    atomicAdd(&st.stats[3], (unsigned long long)(n_kept - fe) * (unsigned long long)dm.L);
  }
}

constexpr int kLayerThreads = 256;

// What both per-layer kernels derive from a sequence's layer budgets.
// 32-bit words of keep bits per (sequence, layer)
__host__ __device__ __forceinline__ size_t kKeepWords(int T) { return ((size_t)T + 31) / 32; }

struct LayerEvent {
  bool event, bad;
  int n, kmin, kmax, P, R, c0, c1;
};

__device__ __forceinline__ LayerEvent layer_event(const DevState& st, const Dims& dm, int b, int seq,
                                                  const int32_t* __restrict__ budget,
                                                  const int32_t* __restrict__ trigger) {
  LayerEvent ev;
  ev.n = st.n_cache[seq];
  ev.kmin = INT_MAX;
  ev.kmax = 0;
  ev.bad = false;
  for (int l = 0; l < dm.L; ++l) {
    const int k = budget[(size_t)b * dm.L + l];
    ev.bad |= k < 1 || k > dm.T;
    ev.kmin = min(ev.kmin, k);
    ev.kmax = max(ev.kmax, k);
  }
  const int trig = trigger ? trigger[b] : ev.kmax;
  ev.event = !ev.bad && ev.n > trig && ev.n > ev.kmin;   // some layer is over its budget
  ev.P = min(st.prefill[seq], ev.n);
  ev.R = ev.bad ? 0 : min(min(dm.recency_cap, ev.kmin / 4), max(0, ev.kmin - ev.P));
  ev.c0 = ev.P;
  ev.c1 = ev.n - ev.R;
  return ev;
}

// Ordered passes of the per-layer kernels: warp w of NW owns the slots
// [w * seg, (w + 1) * seg) and its lanes take 32 consecutive slots at a time
// (coalesced); lane order inside a group of 32 and the warps' totals, scanned
// in shared memory, give each slot its rank.
struct WarpSegment {
  int lo, hi;
};

template <int NW>
__device__ __forceinline__ WarpSegment warp_segment(int n) {
  const int seg = (n + NW * 32 - 1) / (NW * 32) * 32;
  const int lo = min(n, (int)(threadIdx.x >> 5) * seg);
  return WarpSegment{lo, min(n, lo + seg)};
}

// Exclusive prefix over the warps of per-warp totals v (lane 0's value
// counts); *total receives the sum.  wt: NW ints of shared memory.
template <int NW>
__device__ __forceinline__ int warp_base(int v, int* total, int* wt) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) wt[warp] = v;
  __syncthreads();
  int before = 0, all = 0;
  for (int w = 0; w < NW; ++w) {
    before += w < warp ? wt[w] : 0;
    all += wt[w];
  }
  __syncthreads();
  *total = all;
  return before;
}

// Per-layer selection, one CTA per (layer, batch entry): layer l's M_l =
// K_l - P - R best candidates of the union (a radix select on the union's
// candidates), its kept list in its own slot numbering, its new length and
// first moved slot, and one bit per union slot saying whether the layer
// keeps it (a 32-bit word per 32 slots, read by layer_union_kernel).
__global__ void __launch_bounds__(kLayerThreads) layer_keep_kernel(DevState st, Dims dm,
                                                                   const int32_t* __restrict__ seq_ids,
                                                                   const int32_t* __restrict__ budget,
                                                                   const int32_t* __restrict__ trigger,
                                                                   int32_t* __restrict__ kept_out, int kept_stride,
                                                                   int32_t* __restrict__ n_kept_out) {
  pdl_wait();
  pdl_trigger();
  constexpr int NT = kLayerThreads, NW = NT / 32;
  const int l = blockIdx.x, b = blockIdx.y, tid = threadIdx.x, L = dm.L;
  const int lane = tid & 31;
  const unsigned lt = (1u << lane) - 1u;
  const int seq = seq_ids[b];
  if (seq < 0 || seq >= dm.S) {
    if (tid == 0 && l == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  __shared__ RadixShared rs;
  __shared__ int sh_scan[32];
  __shared__ int wt[NW];
  int32_t* nl = st.n_layer + (size_t)seq * L + l;
  int32_t* lf = st.lfirst + (size_t)seq * L + l;
  const LayerEvent ev = layer_event(st, dm, b, seq, budget, trigger);
  if (ev.bad && tid == 0 && l == 0) set_error(st.err, EPIKV_DEV_BUDGET);
  const bool fits = max(ev.kmax, ev.P) <= kept_stride;
  if (ev.event && !fits && tid == 0 && l == 0) set_error(st.err, EPIKV_DEV_KEPT);
  if (!ev.event || !fits) {  // every layer keeps what it holds
    if (tid == 0) {
      *lf = *nl;
      if (n_kept_out) n_kept_out[(size_t)b * L + l] = *nl;
    }
    return;
  }
  const int n = ev.n, c0 = ev.c0, c1 = ev.c1;
  const int M = max(0, budget[(size_t)b * L + l] - ev.P - ev.R);
  const float* __restrict__ sc = st.score[kind_index(st.policy[seq])] + (size_t)seq * dm.T;
  const unsigned long long* __restrict__ mk = st.lmask + (size_t)seq * dm.T;
  uint32_t* __restrict__ keep = st.lkeep + ((size_t)seq * L + l) * kKeepWords(dm.T);
  auto key_at = [&](int i) -> uint32_t { return order_key(sc[i]); };

  // threshold of this layer's M best candidates
  uint32_t theta = 0xFFFFFFFFu;
  int need_eq = 0;
  const bool all = M >= c1 - c0;  // every candidate passes
  const bool sel = M > 0 && !all;
  if (sel) radix_select<NT>(key_at, c0, c1, M, rs, &theta, &need_eq);

  const WarpSegment sg = warp_segment<NW>(n);
  // pass 1: per-warp counts of candidates equal to theta and of held slots
  int ceq = 0, cold = 0;
  for (int i0 = sg.lo; i0 < sg.hi; i0 += 32) {
    const int i = i0 + lane;
    const bool in = i < sg.hi;
    const bool eq = sel && in && i >= c0 && i < c1 && key_at(i) == theta;
    const bool held = in && ((mk[i] >> l) & 1ull);
    ceq += __popc(__ballot_sync(0xffffffffu, eq));
    cold += __popc(__ballot_sync(0xffffffffu, held));
  }
  int n_eq, n_old;
  int q = warp_base<NW>(ceq, &n_eq, wt);
  const int old_base = warp_base<NW>(cold, &n_old, wt);
  // pass 2: the layer's decision per slot (a keep bit, one word per 32 slots), per-warp kept counts
  int cnew = 0;
  for (int i0 = sg.lo; i0 < sg.hi; i0 += 32) {
    const int i = i0 + lane;
    const bool in = i < sg.hi;
    const bool cand = in && i >= c0 && i < c1;
    const bool held = in && ((mk[i] >> l) & 1ull);
    uint32_t key = 0u;
    if (cand && sel) key = key_at(i);
    const bool eq = cand && sel && key == theta;
    const unsigned eb = __ballot_sync(0xffffffffu, eq);
    const int rank = q + __popc(eb & lt);  // among the candidates equal to theta, in slot order
    q += __popc(eb);
    bool k = held;
    if (cand) {
      const bool pass = all || (sel && (key > theta || (eq && rank < need_eq)));
      if (pass && !held) set_error(st.err, EPIKV_DEV_KEPT);  // the layers' caches are not nested
      k = pass && held;
    }
    const unsigned kb = __ballot_sync(0xffffffffu, k);
    if (lane == 0) keep[i0 >> 5] = kb;  // segments start at multiples of 32
    cnew += __popc(kb);
  }
  int n_new;
  int j = warp_base<NW>(cnew, &n_new, wt);
  // pass 3: the kept list, old slot numbers in new slot order
  int32_t* out = kept_out + ((size_t)b * L + l) * kept_stride;
  int o = old_base, fe = INT_MAX;
  for (int i0 = sg.lo; i0 < sg.hi; i0 += 32) {
    const int i = i0 + lane;
    const bool in = i < sg.hi;
    const bool held = in && ((mk[i] >> l) & 1ull);
    const unsigned kb = keep[i0 >> 5];
    const bool k = (kb >> lane) & 1u;
    const unsigned hb = __ballot_sync(0xffffffffu, held);
    if (k) {
      const int my_o = o + __popc(hb & lt), my_j = j + __popc(kb & lt);
      if (my_j < kept_stride) out[my_j] = my_o;
      if (my_o != my_j) fe = min(fe, my_j);
    }
    o += __popc(hb);
    j += __popc(kb);
  }
  fe = block_min<NT>(fe, sh_scan);
  if (tid == 0) {
    if (n_old != *nl) set_error(st.err, EPIKV_DEV_KEPT);  // the masks and the length disagree
    const int f = min(fe, n_new);
    *lf = f;
    *nl = n_new;
    if (n_kept_out) n_kept_out[(size_t)b * L + l] = n_new;
    atomicAdd(&st.stats[3], (unsigned long long)(n_new - f));
  }
}

// The union of the layers after a per-layer selection, one CTA per batch
// entry: each slot's new layer mask (from the keep bits), the kept slots of
// the union (the largest layer's), and the in-place compaction of the slot
// metadata (scores, positions, masks).
__global__ void __launch_bounds__(kSelThreads) layer_union_kernel(DevState st, Dims dm,
                                                                  const int32_t* __restrict__ seq_ids,
                                                                  const int32_t* __restrict__ budget,
                                                                  const int32_t* __restrict__ trigger,
                                                                  int kept_stride, int smem_words) {
  pdl_wait();
  pdl_trigger();
  constexpr int NW = kSelThreads / 32;
  const int b = blockIdx.x, tid = threadIdx.x, L = dm.L;
  const int lane = tid & 31;
  const unsigned lt = (1u << lane) - 1u;
  const int seq = seq_ids[b];
  if (seq < 0 || seq >= dm.S) return;   // reported by layer_keep_kernel
  __shared__ int sh_scan[32];
  __shared__ int wt[NW];
  __shared__ int s_changed;
  const LayerEvent ev = layer_event(st, dm, b, seq, budget, trigger);
  const int n = ev.n;
  if (!ev.event || max(ev.kmax, ev.P) > kept_stride) {
    if (tid == 0) st.first_changed[seq] = n;
    return;
  }
  unsigned long long* __restrict__ mk = st.lmask + (size_t)seq * dm.T;
  unsigned long long* __restrict__ mn = st.lmask_new + (size_t)seq * dm.T;
  const uint32_t* __restrict__ keep = st.lkeep + (size_t)seq * L * kKeepWords(dm.T);
  const size_t kw = kKeepWords(dm.T);
  if (tid == 0) {
    int ch = 0;
    for (int l = 0; l < L; ++l) ch |= st.lfirst[(size_t)seq * L + l] < st.n_layer[(size_t)seq * L + l];
    s_changed = ch;
  }
  // new masks: a warp takes 32 consecutive slots and one keep word per layer
  for (int i0 = (tid >> 5) * 32; i0 < n; i0 += kSelThreads) {
    const int i = i0 + lane;
    unsigned long long m = 0ull;
#pragma unroll 8
    for (int l = 0; l < L; ++l) m |= (unsigned long long)((keep[l * kw + (i0 >> 5)] >> lane) & 1u) << l;
    if (i < n) mn[i] = m;
  }
  __syncthreads();
  const WarpSegment sg = warp_segment<NW>(n);
  int cu = 0;
  for (int i0 = sg.lo; i0 < sg.hi; i0 += 32) {
    const int i = i0 + lane;
    cu += __popc(__ballot_sync(0xffffffffu, i < sg.hi && mn[i] != 0ull));
  }
  int n_union;
  int o = warp_base<NW>(cu, &n_union, wt);
  int32_t* mkept = st.mkept + (size_t)seq * dm.T;
  int fe = INT_MAX;
  for (int i0 = sg.lo; i0 < sg.hi; i0 += 32) {
    const int i = i0 + lane;
    const bool k = i < sg.hi && mn[i] != 0ull;
    const unsigned kb = __ballot_sync(0xffffffffu, k);
    if (k) {
      const int my_o = o + __popc(kb & lt);
      mkept[my_o] = i;
      if (my_o != i) fe = min(fe, my_o);
    }
    o += __popc(kb);
  }
  fe = min(block_min(fe, sh_scan), n_union);
  __syncthreads();  // the union's kept list is visible to the whole block
  extern __shared__ uint32_t stage[];
  compact_metadata(st, dm, seq, mkept, fe, n_union, stage, smem_words);
  // every new mask lands in its slot (the slots before fe did not move)
  for (int j = tid; j < n_union; j += kSelThreads) mk[j] = mn[mkept[j]];
  if (tid == 0) {
    st.n_cache[seq] = n_union;
    st.first_changed[seq] = s_changed ? 0 : n_union;
    atomicAdd(&st.stats[1], 1ull);
    atomicAdd(&st.stats[2], (unsigned long long)(n_union - fe));
  }
}

// Candidate keys staged in shared memory: caches of up to kSelStagedMax slots.
// The same memory then stages the slot metadata's compaction: one round for
// every kind's score and the position of each slot, when it fits.
constexpr int kSelStagedMax = 48 * 1024;  // 192 KiB of u32 words
static int sel_staged_cap(const Dims& dm) { return dm.T <= kSelStagedMax ? dm.T : 0; }
static int sel_smem_words(const Dims& dm) {
  const int64_t ncol = __builtin_popcount((unsigned)dm.kinds) + 1;  // metadata columns
  const int64_t meta = ncol * dm.T;
  int64_t w = meta > sel_staged_cap(dm) ? meta : sel_staged_cap(dm);
  const int64_t fused = ((int64_t)dm.T + 3) / 4 * 4 + (ncol + 1) * dm.T;  // keys, every column, the kept list
  if (ncol <= kFusedCols && fused <= kSelStagedMax && fused > w) w = fused;
  return (int)(w < kSelStagedMax ? w : kSelStagedMax);
}
static size_t sel_smem(const Dims& dm) { return (size_t)sel_smem_words(dm) * sizeof(uint32_t); }

cudaError_t select_prepare() {
  const int mx = kSelStagedMax * (int)sizeof(uint32_t);
  cudaError_t e = cudaFuncSetAttribute(select_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(select_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  if (e == cudaSuccess) e = cudaFuncSetAttribute(layer_union_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, mx);
  return e;
}

cudaError_t launch_select(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                          const int32_t* budget, const int32_t* trigger, int32_t* kept, int kept_stride,
                          int32_t* n_kept, cudaStream_t stream, int* launches) {
  if (n_seq == 0) return cudaSuccess;
  const size_t smem = sel_smem(dm);
  const int words = sel_smem_words(dm);
  if (dm.layer_budgets) {
    pdl_launch(layer_keep_kernel, dim3(dm.L, n_seq), kLayerThreads, 0, stream, st, dm, seq_ids, budget, trigger,
               kept, kept_stride, n_kept);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    ++*launches;
    pdl_launch(layer_union_kernel, n_seq, kSelThreads, smem, stream, st, dm, seq_ids, budget, trigger, kept_stride,
               words);
  } else if (dm.select_chunk > 1) {
    pdl_launch(select_kernel<true>, n_seq, kSelThreads, smem, stream, st, dm, seq_ids, budget, trigger, kept,
               kept_stride, n_kept, sel_staged_cap(dm), words);
  } else if (dm.T > EPIKV_SEL_CLUSTER_MIN) {
    pdl_launch(select_cluster_kernel, n_seq * kCluCtas, kCluThreads, (size_t)kCluStageWords * sizeof(uint32_t),
               stream, st, dm, seq_ids, budget, trigger, kept, kept_stride, n_kept);
  } else {
    pdl_launch(select_kernel<false>, n_seq, kSelThreads, smem, stream, st, dm, seq_ids, budget, trigger, kept,
               kept_stride, n_kept, sel_staged_cap(dm), words);
  }
  ++*launches;
  return cudaGetLastError();
}

}  // namespace epikv
