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
// safe in increasing order because kept[i] >= i.
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
// holding it.  select_layers_kernel runs one radix select per distinct M_l =
// K_l - P - R over the union's candidates (largest M first), gives each
// candidate the mask of the layers whose threshold it passes, and turns the
// old and new masks into one kept list per layer in that layer's own slot
// numbering (a block scan per layer), then compacts the union's metadata.
#include "common.cuh"
#include "kernels.h"

namespace epikv {

constexpr int kSelThreads = 1024;

__device__ __forceinline__ uint32_t order_key(float f) {
  if (f != f) return 0u;          // NaN below every number
  if (f == 0.0f) f = 0.0f;        // -0 == +0
  const uint32_t b = __float_as_uint(f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// Exclusive prefix sum over the block; *total receives the sum.
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
    int w = lane < (kSelThreads / 32) ? sh[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    sh[lane] = w;  // inclusive warp totals
  }
  __syncthreads();
  const int before = (warp > 0 ? sh[warp - 1] : 0) + x - v;
  *total = sh[kSelThreads / 32 - 1];
  __syncthreads();
  return before;
}

__device__ __forceinline__ int block_min(int v, int* sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = min(v, __shfl_xor_sync(0xffffffffu, v, o));
  if (lane == 0) sh[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int w = lane < (kSelThreads / 32) ? sh[lane] : INT_MAX;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) w = min(w, __shfl_xor_sync(0xffffffffu, w, o));
    if (lane == 0) sh[0] = w;
  }
  __syncthreads();
  const int r = sh[0];
  __syncthreads();
  return r;
}

struct RadixShared {
  uint32_t hist[256];
  uint32_t prefix, mask, remaining;
};

// The M-th largest key_at(i) over i in [c0, c1), 0 < M <= c1 - c0, by a
// 4-pass 8-bit radix select: *theta is that key and *need_eq the number of
// keys equal to it that belong to the M largest (the lowest slots first).
// Every thread of the block calls it.
template <typename KeyAt>
__device__ __forceinline__ void radix_select(const KeyAt& key_at, int c0, int c1, int M, RadixShared& rs,
                                             uint32_t* theta, int* need_eq) {
  const int tid = threadIdx.x;
  __syncthreads();  // every thread has read the previous call's result
  if (tid == 0) {
    rs.prefix = 0u;
    rs.mask = 0u;
    rs.remaining = (uint32_t)M;
  }
  for (int shift = 24; shift >= 0; shift -= 8) {
    if (tid < 256) rs.hist[tid] = 0u;
    __syncthreads();
    const uint32_t prefix = rs.prefix, mask = rs.mask;
    for (int i = c0 + tid; i < c1; i += kSelThreads) {
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
}

template <bool kChunked>
__global__ void __launch_bounds__(kSelThreads) select_kernel(DevState st, Dims dm,
                                                             const int32_t* __restrict__ seq_ids,
                                                             const int32_t* __restrict__ budget,
                                                             const int32_t* __restrict__ trigger,
                                                             int32_t* __restrict__ kept_out, int kept_stride,
                                                             int32_t* __restrict__ n_kept_out) {
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
  auto key_at = [&](int i) -> uint32_t { return kChunked ? ck[i] : order_key(sc[i]); };

  __shared__ RadixShared rs;
  __shared__ int sh_scan[32];

  // ---- radix select of the M-th largest key among the candidates
  uint32_t theta = 0xFFFFFFFFu;
  int need_eq = 0;
  if (M > 0) radix_select(key_at, c0, c1, M, rs, &theta, &need_eq);

  // ---- ordered scans over contiguous per-thread slot ranges
  const int per = (n + kSelThreads - 1) / kSelThreads;
  const int a = min(n, tid * per), e = min(n, a + per);
  int eq_local = 0;
  for (int i = max(a, c0); i < min(e, c1); ++i) eq_local += (key_at(i) == theta);
  int tot;
  const int eq_base = block_exclusive_scan(eq_local, &tot, sh_scan);

  int keep_local = 0, first_ev = INT_MAX;
  {
    int eqs = eq_base;
    for (int i = a; i < e; ++i) {
      bool keep = (i < c0) || (i >= c1);
      if (!keep) {
        const uint32_t k = key_at(i);
        keep = k > theta || (k == theta && eqs++ < need_eq);
      }
      if (keep) ++keep_local; else first_ev = min(first_ev, i);
    }
  }
  int n_kept;
  const int keep_base = block_exclusive_scan(keep_local, &n_kept, sh_scan);
  {
    int eqs = eq_base, o = keep_base;
    for (int i = a; i < e; ++i) {
      bool keep = (i < c0) || (i >= c1);
      if (!keep) {
        const uint32_t k = key_at(i);
        keep = k > theta || (k == theta && eqs++ < need_eq);
      }
      if (keep) out[o++] = i;
    }
  }
  const int fe = min(block_min(first_ev, sh_scan), n_kept);
  __syncthreads();  // kept list visible to the whole block

  // ---- compact slot metadata in place (kept[i] >= i, increasing i)
  int32_t* ps = st.pos + (size_t)seq * dm.T;
  for (int j0 = fe; j0 < n_kept; j0 += kSelThreads) {
    const int j = j0 + tid;
    float v[kNumKinds];
    int32_t p = 0;
    if (j < n_kept) {
      const int src = out[j];
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
  if (tid == 0) {
    st.n_cache[seq] = n_kept;
    st.first_changed[seq] = fe;
    if (n_kept_out) n_kept_out[b] = n_kept;
    atomicAdd(&st.stats[1], 1ull);
    atomicAdd(&st.stats[2], (unsigned long long)(n_kept - fe));
    atomicAdd(&st.stats[3], (unsigned long long)(n_kept - fe) * (unsigned long long)dm.L);
  }
}

constexpr int kMaxLayers = 64;

__global__ void __launch_bounds__(kSelThreads) select_layers_kernel(DevState st, Dims dm,
                                                                    const int32_t* __restrict__ seq_ids,
                                                                    const int32_t* __restrict__ budget,
                                                                    const int32_t* __restrict__ trigger,
                                                                    int32_t* __restrict__ kept_out, int kept_stride,
                                                                    int32_t* __restrict__ n_kept_out) {
  const int b = blockIdx.x, tid = threadIdx.x, L = dm.L;
  const int seq = seq_ids[b];
  if (seq < 0 || seq >= dm.S) {
    if (tid == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  __shared__ int sK[kMaxLayers];
  __shared__ int s_bad, s_changed, s_ng;
  __shared__ int s_gM[kMaxLayers];
  __shared__ unsigned long long s_gbits[kMaxLayers];
  __shared__ RadixShared rs;
  __shared__ int sh_scan[32];
  int32_t* nl = st.n_layer + (size_t)seq * L;
  int32_t* lf = st.lfirst + (size_t)seq * L;
  const int n = st.n_cache[seq];
  if (tid == 0) {
    s_bad = 0;
    s_changed = 0;
  }
  __syncthreads();
  if (tid < L) {
    const int k = budget[(size_t)b * L + tid];
    sK[tid] = k;
    if (k < 1 || k > dm.T) atomicOr(&s_bad, 1);
  }
  __syncthreads();
  // no event: every layer keeps what it holds
  auto keep_all = [&]() {
    for (int l = tid; l < L; l += kSelThreads) {
      lf[l] = nl[l];
      if (n_kept_out) n_kept_out[(size_t)b * L + l] = nl[l];
    }
    if (tid == 0) st.first_changed[seq] = n;
  };
  if (s_bad) {
    if (tid == 0) set_error(st.err, EPIKV_DEV_BUDGET);
    keep_all();
    return;
  }
  int kmin = INT_MAX, kmax = 0;
  for (int l = 0; l < L; ++l) {
    kmin = min(kmin, sK[l]);
    kmax = max(kmax, sK[l]);
  }
  const int trig = trigger ? trigger[b] : kmax;
  if (n <= trig || n <= kmin) {  // no layer is over its budget, or no event yet
    keep_all();
    return;
  }
  const int P = min(st.prefill[seq], n);
  const int R = min(min(dm.recency_cap, kmin / 4), max(0, kmin - P));
  const int c0 = P, c1 = n - R;  // the union's candidates [c0, c1)
  if (max(kmax, P) > kept_stride) {
    if (tid == 0) set_error(st.err, EPIKV_DEV_KEPT);
    keep_all();
    return;
  }
  const float* __restrict__ sc = st.score[kind_index(st.policy[seq])] + (size_t)seq * dm.T;
  unsigned long long* __restrict__ mk = st.lmask + (size_t)seq * dm.T;
  unsigned long long* __restrict__ mn = st.lmask_new + (size_t)seq * dm.T;
  auto key_at = [&](int i) -> uint32_t { return order_key(sc[i]); };

  // ---- layers grouped by equal M_l, largest M first; s_gbits[g] holds the
  // layers of groups 0..g (those that keep a candidate group g keeps)
  if (tid == 0) {
    int ord[kMaxLayers];
    for (int l = 0; l < L; ++l) {
      const int m = max(0, sK[l] - P - R);
      int j = l;
      while (j > 0 && max(0, sK[ord[j - 1]] - P - R) < m) {
        ord[j] = ord[j - 1];
        --j;
      }
      ord[j] = l;
    }
    int ng = 0;
    unsigned long long bits = 0ull;
    for (int j = 0; j < L; ++j) {
      const int m = max(0, sK[ord[j]] - P - R);
      if (j > 0 && m != s_gM[ng - 1]) ++ng;
      if (j == 0) ng = 1;
      s_gM[ng - 1] = m;
      bits |= 1ull << ord[j];
      s_gbits[ng - 1] = bits;
    }
    s_ng = ng;
  }
  // protected slots keep their layers; candidates start with none
  for (int i = tid; i < n; i += kSelThreads) mn[i] = (i < c0 || i >= c1) ? mk[i] : 0ull;
  __syncthreads();

  const int ncand = c1 - c0;
  const int per = (n + kSelThreads - 1) / kSelThreads;
  const int a = min(n, tid * per), e = min(n, a + per);
  for (int g = 0; g < s_ng; ++g) {
    const int M = s_gM[g];
    const unsigned long long bits = s_gbits[g];
    if (M <= 0) break;  // this group and the smaller ones keep no candidate
    if (M >= ncand) {   // every candidate passes
      for (int i = c0 + tid; i < c1; i += kSelThreads) mn[i] = bits;
      __syncthreads();
      continue;
    }
    uint32_t theta;
    int need_eq;
    radix_select(key_at, c0, c1, M, rs, &theta, &need_eq);
    int eq_local = 0;
    for (int i = max(a, c0); i < min(e, c1); ++i) eq_local += (key_at(i) == theta);
    int tot;
    int eqs = block_exclusive_scan(eq_local, &tot, sh_scan);
    for (int i = max(a, c0); i < min(e, c1); ++i) {
      const uint32_t k = key_at(i);
      if (k > theta || (k == theta && eqs++ < need_eq)) mn[i] = bits;
    }
    __syncthreads();
  }
  // a layer keeps only tokens it holds (true by the nesting; checked)
  for (int i = c0 + tid; i < c1; i += kSelThreads) {
    const unsigned long long nm = mn[i], om = mk[i];
    if (nm & ~om) set_error(st.err, EPIKV_DEV_KEPT);
    mn[i] = nm & om;
  }
  __syncthreads();

  // ---- one kept list per layer, in that layer's slot numbering
  unsigned long long moved = 0ull;
  for (int l = 0; l < L; ++l) {
    int co = 0, cn = 0;
    for (int i = a; i < e; ++i) {
      co += (int)((mk[i] >> l) & 1ull);
      cn += (int)((mn[i] >> l) & 1ull);
    }
    int n_old, n_new;
    int o = block_exclusive_scan(co, &n_old, sh_scan);
    int j = block_exclusive_scan(cn, &n_new, sh_scan);
    int32_t* out = kept_out + ((size_t)b * L + l) * kept_stride;
    int fe = INT_MAX;
    for (int i = a; i < e; ++i) {
      if ((mn[i] >> l) & 1ull) {
        if (j < kept_stride) out[j] = o;
        if (o != j) fe = min(fe, j);
        ++j;
      }
      if ((mk[i] >> l) & 1ull) ++o;
    }
    fe = block_min(fe, sh_scan);
    if (tid == 0) {
      if (n_old != nl[l]) set_error(st.err, EPIKV_DEV_KEPT);  // masks and length disagree
      const int f = min(fe, n_new);
      lf[l] = f;
      nl[l] = n_new;
      if (n_kept_out) n_kept_out[(size_t)b * L + l] = n_new;
      moved += (unsigned long long)(n_new - f);
      if (f < n_new) s_changed = 1;
    }
  }

  // ---- the union's kept slots (any layer holds them), then its metadata
  int32_t* mkept = st.mkept + (size_t)seq * dm.T;
  int cu = 0;
  for (int i = a; i < e; ++i) cu += mn[i] != 0ull;
  int n_union;
  int o = block_exclusive_scan(cu, &n_union, sh_scan);
  int fe = INT_MAX;
  for (int i = a; i < e; ++i)
    if (mn[i] != 0ull) {
      mkept[o] = i;
      if (o != i) fe = min(fe, o);
      ++o;
    }
  fe = min(block_min(fe, sh_scan), n_union);
  __syncthreads();  // the union's kept list is visible to the whole block
  int32_t* ps = st.pos + (size_t)seq * dm.T;
  for (int j0 = fe; j0 < n_union; j0 += kSelThreads) {
    const int j = j0 + tid;
    float v[kNumKinds];
    int32_t p = 0;
    if (j < n_union) {
      const int src = mkept[j];
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k) v[k] = st.score[k] ? st.score[k][(size_t)seq * dm.T + src] : 0.f;
      p = ps[src];
    }
    __syncthreads();
    if (j < n_union) {
#pragma unroll
      for (int k = 0; k < kNumKinds; ++k)
        if (st.score[k]) st.score[k][(size_t)seq * dm.T + j] = v[k];
      ps[j] = p;
    }
    __syncthreads();
  }
  // every new mask lands in its slot (the ones before fe did not move)
  for (int j = tid; j < n_union; j += kSelThreads) mk[j] = mn[mkept[j]];
  __syncthreads();
  if (tid == 0) {
    st.n_cache[seq] = n_union;
    st.first_changed[seq] = s_changed ? 0 : n_union;
    atomicAdd(&st.stats[1], 1ull);
    atomicAdd(&st.stats[2], (unsigned long long)(n_union - fe));
    atomicAdd(&st.stats[3], moved);
  }
}

cudaError_t launch_select(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                          const int32_t* budget, const int32_t* trigger, int32_t* kept, int kept_stride,
                          int32_t* n_kept, cudaStream_t stream, int* launches) {
  if (n_seq == 0) return cudaSuccess;
  if (dm.layer_budgets)
    select_layers_kernel<<<n_seq, kSelThreads, 0, stream>>>(st, dm, seq_ids, budget, trigger, kept, kept_stride,
                                                            n_kept);
  else if (dm.select_chunk > 1)
    select_kernel<true><<<n_seq, kSelThreads, 0, stream>>>(st, dm, seq_ids, budget, trigger, kept, kept_stride,
                                                           n_kept);
  else
    select_kernel<false><<<n_seq, kSelThreads, 0, stream>>>(st, dm, seq_ids, budget, trigger, kept, kept_stride,
                                                            n_kept);
  ++*launches;
  return cudaGetLastError();
}

}  // namespace epikv
