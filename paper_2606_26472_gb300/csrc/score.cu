// Scoring kernels of the EpiKV hot path.
//
//   bandz_g_kernel         g_l(t) = ||h_l(t) - h_l(t-1)||_2 of every new token
//                          and band layer (Sec. 3.2, Eq. 1), streamed from the
//                          bf16 rows with 16-byte loads, fp32 accumulation.
//   lagkv_partial_kernel   Lag-KV (Sec. 3.3): each new token's K or V row of one
//                          layer, normalised by the previous chunk's per-channel
//                          range; population variance over the head dimension,
//                          summed over heads.  Keeps the running chunk ranges.
//   score_finalize_kernel  causal rolling z-score per band layer and the band
//                          combination (Eq. 3, Fig. 1); Lag-KV u(t) and its
//                          rolling mean; writes the frozen score and position of
//                          every new slot and commits the sequence's counters.
//
// Every result is independent of how a trace is split into calls: g values
// and u values are computed from the same bytes in the same order whether the
// previous row comes from the call or from the saved state, and the window
// reductions run over positions in a fixed lane order.
#include <type_traits>

#include "common.cuh"
#include "kernels.h"

namespace epikv {

#ifndef EPIKV_G_UNROLL
#define EPIKV_G_UNROLL 2  // tokens whose rows are loaded together (measured best: 2)
#endif
constexpr int kGThreads = 256;
constexpr int kGUnroll = EPIKV_G_UNROLL;
constexpr int kMaxTokPerCta = 16;

struct BandRows {
  const __nv_bfloat16* p[kMaxBand];
};

// Persistent grid; block: 256 threads.  The rows of the call, flattened as
// r = band * total_new + packed_row, are split into gridDim.x equal
// contiguous shares, so every CTA streams the same number of rows.  A CTA
// walks its share in runs that stay inside one (band layer, batch entry),
// 16 tokens at most; the previous row of a run's first token is the last row
// of the run before it when they are consecutive, else it is loaded (from
// the saved h_prev for a sequence's first new token).
template <int VPT>
#ifndef EPIKV_G_MINB
#define EPIKV_G_MINB 0  // 0: by register need
#endif
__global__ void __launch_bounds__(kGThreads, (EPIKV_G_MINB > 0 ? EPIKV_G_MINB : VPT * kGUnroll >= 16 ? 2 : 4)) bandz_g_kernel(DevState st, Dims dm, BandRows rows,
                                                            int64_t row_stride,
                                                            const int32_t* __restrict__ seq_ids,
                                                            const int32_t* __restrict__ cu_new, int n_seq,
                                                            int max_new) {
  pdl_wait();
  pdl_trigger();
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // the whole batch must be well formed, else nothing is read
  __shared__ int bad;
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int b = tid; b < n_seq; b += kGThreads) {
    const int seq = seq_ids[b], n = cu_new[b + 1] - cu_new[b];
    if (seq < 0 || seq >= dm.S || n < 0 || n > max_new || cu_new[0] != 0) bad = 1;
  }
  __syncthreads();
  if (bad) {
    if (tid == 0 && blockIdx.x == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  const int nb = dm.nA + dm.nB;
  const int total = cu_new[n_seq];
  const int64_t R = (int64_t)nb * total;
  int64_t r = R * blockIdx.x / gridDim.x;
  const int64_t r_end = R * (blockIdx.x + 1) / gridDim.x;
  if (r >= r_end) return;
  const int VR = dm.D >> 3;  // 16-byte vectors per row
  __shared__ float red[kMaxTokPerCta][kGThreads / 32];  // per token of a run, per warp

  int band = (int)(r / total), row = (int)(r - (int64_t)band * total);
  int b = 0;  // batch entry holding `row` (largest b with cu_new[b] <= row and a token)
  {
    int lo = 0, hi = n_seq - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) >> 1;
      if (cu_new[mid] <= row) lo = mid; else hi = mid - 1;
    }
    b = lo;
    while (cu_new[b + 1] <= row) ++b;  // skip empty entries
  }
  uint4 prev[VPT];
  int prev_band = -1, prev_row = -1;  // what `prev` holds
  while (r < r_end) {
    const int r0 = cu_new[b], n_new = cu_new[b + 1] - r0;
    const int seq = seq_ids[b];
    const int t0 = row - r0;
    const int len = (int)min((int64_t)min(kMaxTokPerCta, n_new - t0), r_end - r);
    const int t1 = t0 + len;
    const int p0 = st.n_seen[seq];
    const int par = st.hp_parity[seq];
    const __nv_bfloat16* base = rows.p[band];
    if (!(prev_band == band && prev_row == row - 1 && t0 > 0)) {
      const __nv_bfloat16* prow = t0 == 0 ? st.h_prev + ((size_t)(seq * 2 + par) * nb + band) * dm.D
                                          : base + (int64_t)(row - 1) * row_stride;
#pragma unroll
      for (int k = 0; k < VPT; ++k) {
        const int v = tid + k * kGThreads;
        prev[k] = v < VR ? ld_stream16(prow + v * 8) : make_uint4(0, 0, 0, 0);
      }
    }
    for (int t = t0; t < t1; t += kGUnroll) {
      uint4 cur[kGUnroll][VPT];
#pragma unroll
      for (int u = 0; u < kGUnroll; ++u) {
        const __nv_bfloat16* rp = base + (int64_t)(r0 + t + u) * row_stride;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
          const int v = tid + k * kGThreads;
          cur[u][k] = (t + u < t1 && v < VR) ? ld_stream16(rp + v * 8) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int u = 0; u < kGUnroll; ++u) {
        float acc = 0.f;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
          float c[8], p[8];
          unpack8(cur[u][k], c);
          unpack8(u == 0 ? prev[k] : cur[u - 1][k], p);
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float dlt = c[e] - p[e];
            acc = fmaf(dlt, dlt, acc);
          }
        }
        acc = warp_sum(acc);
        if (lane == 0 && t + u < t1) red[t - t0 + u][warp] = acc;
      }
      // the last valid row of this group is the previous row of the next group
      const int last = min(kGUnroll, t1 - t) - 1;
#pragma unroll
      for (int u = 0; u < kGUnroll; ++u)
        if (u == last) {
#pragma unroll
          for (int k = 0; k < VPT; ++k) prev[k] = cur[u][k];
        }
    }
    __syncthreads();
    if (tid < len) {
      float sum = 0.f;
#pragma unroll
      for (int w = 0; w < kGThreads / 32; ++w) sum += red[tid][w];
      const int pos = p0 + t0 + tid;
      if (pos >= 1) st.g_ring[((size_t)seq * nb + band) * dm.G + (pos & (dm.G - 1))] = sqrtf(sum);
    }
    if (t1 == n_new) {  // the sequence's last new row of this band is the next call's previous row
      __nv_bfloat16* hp_wr = st.h_prev + ((size_t)(seq * 2 + (par ^ 1)) * nb + band) * dm.D;
#pragma unroll
      for (int k = 0; k < VPT; ++k) {
        const int v = tid + k * kGThreads;
        if (v < VR) *reinterpret_cast<uint4*>(hp_wr + v * 8) = prev[k];
      }
    }
    __syncthreads();  // red is reused by the next run
    prev_band = band;
    prev_row = row + len - 1;
    r += len;
    row += len;
    if (row == total) {
      row = 0;
      ++band;
      b = 0;
    }
    while (b < n_seq && cu_new[b + 1] <= row) ++b;
  }
}

#ifndef EPIKV_LAG_SEG
#define EPIKV_LAG_SEG 8
#endif
#ifndef EPIKV_LAG_MINB
#define EPIKV_LAG_MINB 3  // with EPIKV_LAG_MAXREG 0: registers capped at 80
#endif
#ifndef EPIKV_LAG_PF
#define EPIKV_LAG_PF 1  // measured: 1 segment ahead 110 us, none 115 us, 2 ahead 119 us
#endif
constexpr int kLagSeg = EPIKV_LAG_SEG;  // tokens per segment (never crosses a chunk boundary)
constexpr int kLagPf = EPIKV_LAG_PF;    // a row is prefetched into L2 this many segments ahead
constexpr int kLagOffs = 256;   // slot offsets looked up per group of tokens

// Fire-and-forget bulk prefetch of [p, p + bytes) into L2 (p 16-byte aligned,
// bytes a multiple of 16).
__device__ __forceinline__ void prefetch_l2_bulk(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" :: "l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ uint32_t bf16x2_min(uint32_t a, uint32_t b) {
  __nv_bfloat162 r = __hmin2(*reinterpret_cast<__nv_bfloat162*>(&a), *reinterpret_cast<__nv_bfloat162*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}
__device__ __forceinline__ uint32_t bf16x2_max(uint32_t a, uint32_t b) {
  __nv_bfloat162 r = __hmax2(*reinterpret_cast<__nv_bfloat162*>(&a), *reinterpret_cast<__nv_bfloat162*>(&b));
  return *reinterpret_cast<uint32_t*>(&r);
}
__device__ __forceinline__ uint4 q_min(const uint4& a, const uint4& b) {
  return make_uint4(bf16x2_min(a.x, b.x), bf16x2_min(a.y, b.y), bf16x2_min(a.z, b.z), bf16x2_min(a.w, b.w));
}
__device__ __forceinline__ uint4 q_max(const uint4& a, const uint4& b) {
  return make_uint4(bf16x2_max(a.x, b.x), bf16x2_max(a.y, b.y), bf16x2_max(a.z, b.z), bf16x2_max(a.w, b.w));
}

// ---- packed fp32 pairs: Blackwell's f32x2 arithmetic, two channels per instruction
typedef unsigned long long f32x2;

__device__ __forceinline__ f32x2 f2_pack(float lo, float hi) {
  f32x2 d;
  asm("mov.b64 %0, {%1, %2};" : "=l"(d) : "f"(lo), "f"(hi));
  return d;
}
__device__ __forceinline__ float f2_lo(f32x2 v) { return __uint_as_float((unsigned)(v & 0xffffffffull)); }
__device__ __forceinline__ float f2_hi(f32x2 v) { return __uint_as_float((unsigned)(v >> 32)); }
__device__ __forceinline__ f32x2 f2_fma(f32x2 a, f32x2 b, f32x2 c) {
  f32x2 d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}
__device__ __forceinline__ f32x2 f2_add(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("add.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
__device__ __forceinline__ f32x2 f2_mul(f32x2 a, f32x2 b) {
  f32x2 d;
  asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
  return d;
}
// the two bf16 channels of a 32-bit word as an fp32 pair (exact)
__device__ __forceinline__ f32x2 bf16x2_to_f2(uint32_t w) { return f2_pack(bf16_lo(w), bf16_hi(w)); }

// The previous chunk's range as a per-channel affine map y = x * a + c with
// a = 1 / (max - min + eps) and c = -min * a - 1/2, so that y = x~ - 1/2 for
// the range-normalised x~ (one fused multiply-add per channel).
__device__ __forceinline__ void prev_affine(const uint4& pmn, const uint4& pmx, float eps, f32x2 (&a)[4],
                                            f32x2 (&c)[4]) {
  float mn[8], mx[8], inv[8], bias[8];
  unpack8(pmn, mn);
  unpack8(pmx, mx);
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    inv[e] = __frcp_rn(mx[e] - mn[e] + eps);   // the correctly rounded reciprocal (as 1.f / x)
    bias[e] = fmaf(-mn[e], inv[e], -0.5f);
  }
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    a[p] = f2_pack(inv[2 * p], inv[2 * p + 1]);
    c[p] = f2_pack(bias[2 * p], bias[2 * p + 1]);
  }
}

// Sums of y and y^2 over one thread's 8 channels of a token row.
__device__ __forceinline__ void lag_moments(const uint4& x, const f32x2 (&a)[4], const f32x2 (&c)[4], float& s1,
                                            float& s2) {
  const f32x2 y0 = f2_fma(bf16x2_to_f2(x.x), a[0], c[0]);
  const f32x2 y1 = f2_fma(bf16x2_to_f2(x.y), a[1], c[1]);
  const f32x2 y2 = f2_fma(bf16x2_to_f2(x.z), a[2], c[2]);
  const f32x2 y3 = f2_fma(bf16x2_to_f2(x.w), a[3], c[3]);
  const f32x2 t = f2_add(f2_add(y0, y1), f2_add(y2, y3));
  f32x2 u = f2_mul(y0, y0);
  u = f2_fma(y1, y1, u);
  u = f2_fma(y2, y2, u);
  u = f2_fma(y3, y3, u);
  s1 = f2_lo(t) + f2_hi(t);
  s2 = f2_lo(u) + f2_hi(u);
}

// Transposed sum over the O*2 lanes of a group: every level halves the values
// a lane keeps and sends the other half to its partner, so NV values cost
// NV - 1 shuffles in all instead of one butterfly of log2(lanes) shuffles per
// value.  With lanes <= NV, value k + (NV / lanes) * (lane % lanes) ends in
// v[k]; with more lanes than values, value (lane % lanes) / (lanes / NV) ends
// in v[0].
template <int O, int C, int NV>
__device__ __forceinline__ void transpose_sum(float (&v)[NV], int lane) {
  if constexpr (O >= 1) {
    if constexpr (C > 1) {
      const bool up = lane & O;
#pragma unroll
      for (int k = 0; k < C / 2; ++k) {
        const float send = up ? v[k] : v[k + C / 2];
        const float keep = up ? v[k + C / 2] : v[k];
        v[k] = keep + __shfl_xor_sync(0xffffffffu, send, O);
      }
      transpose_sum<O / 2, C / 2, NV>(v, lane);
    } else {
      v[0] += __shfl_xor_sync(0xffffffffu, v[0], O);
      transpose_sum<O / 2, 1, NV>(v, lane);
    }
  }
}

// grid: (2L (layer, K|V), batch entries); block: max(32, H*d/8) threads;
// LH = d/8 consecutive lanes own one head, 8 channels each.
//
// Tokens are taken in segments that stay inside one chunk: every token of a
// segment is normalised with the same previous-chunk range, so the segment's
// reductions are independent of one another.  Chunk ranges (min, max) are
// bf16 values and are kept packed (exact).  The variance of a token's head
// is taken from the moments of y = x~ - 1/2 (x~ in [0, 1] inside the range),
// computed two channels per instruction (f32x2); the segment's 2 x 8 moments
// are summed over the head's lanes by one transposed reduction into shared
// memory, where a thread per token forms each head's variance.
//
// The stream's work is lag_stream, which the one-token decode kernel
// (token_kernel) runs unchanged for its K/V CTAs.
// SEG is the longest segment: kLagSeg, or 1 for one-token calls (fewer
// registers; the reductions pair lanes in the same order either way, so the
// sums are the same bit for bit).  With HALF, each half of a 256-thread
// block runs its own stream (K in the first half, V in the second; H*d/8 <=
// 128), with its own shared memory.
// KINDS: 0 = whichever K/V kinds the context computes (runtime flags); 1 =
// the normalised kinds only; 2 = the raw kinds only; 3 = both (compile-time,
// so a kernel instance holds only the registers its kinds need).
#ifndef EPIKV_TOKEN_OWN_OFFSET
#define EPIKV_TOKEN_OWN_OFFSET 1  // 0: one-token calls also look the row up through shared memory
#endif
template <int LH, int SEG = kLagSeg, bool HALF = false, int KINDS = 0>
__device__ __forceinline__ void lag_stream(const DevState& st, const Dims& dm, const KvDev& kv, int seq,
                                           int n_new, int layer, int kvk, int nc0) {
  const int stream = layer * 2 + kvk;  // this stream's column of the per-token partials
  const int tid = HALF ? (int)(threadIdx.x & 127) : (int)threadIdx.x;
  const int nthr = HALF ? 128 : (int)blockDim.x;
  const int half = HALF ? kvk : 0;
  const int h = tid / LH, q = tid % LH;
  const bool active = h < dm.H;
  const int hd = dm.H * dm.d;
  const int p0 = st.n_seen[seq];
  const int ch = h * dm.d + q * 8;  // first channel of this thread within the token row
  const bool need_norm = KINDS ? (KINDS & 1) != 0 : (dm.kinds & kNormKinds) != 0;   // uniform across the grid
  const bool need_raw = KINDS ? (KINDS & 2) != 0 : (dm.kinds & kRawKinds) != 0;
  __nv_bfloat16* rng = need_norm ? st.lag_rng + ((((size_t)seq * dm.L + layer) * 2 + kvk) * 4) * hd : nullptr;

  // the previous chunk's range lives on only as its affine map; it is written
  // back as soon as a chunk completes, the running range at the end
  uint4 cmn = make_uint4(0, 0, 0, 0), cmx = cmn;
  f32x2 na[4], nc[4];
  {
    uint4 pmn = cmn, pmx = cmn;
    if (active && need_norm) {
      pmn = *reinterpret_cast<const uint4*>(rng + 0 * hd + ch);
      pmx = *reinterpret_cast<const uint4*>(rng + 1 * hd + ch);
      cmn = *reinterpret_cast<const uint4*>(rng + 2 * hd + ch);
      cmx = *reinterpret_cast<const uint4*>(rng + 3 * hd + ch);
    }
    prev_affine(pmn, pmx, dm.lag_eps, na, nc);
  }

  const float inv_d = 1.f / (float)dm.d;
  const char* kvbase = kvk ? kv.base[1] : kv.base[0];  // a select: no local copy of the parameter struct
  const char* kvb_ch = kvbase + (int64_t)ch * 2;       // this thread's first channel in a row at offset 0
  __shared__ int64_t soff_s[HALF ? 2 : 1][kLagOffs];
  constexpr int NV = 2 * SEG;      // moments of a segment: (sum y, sum y^2) per token
  __shared__ float red_s[HALF ? 2 : 1][2][32][NV];  // [half][segment parity][head][moment]; the host admits H <= 32
  __shared__ float hr_s[HALF ? 2 : 1][2][SEG][32];  // raw variances, same layout
  int64_t* soff = soff_s[half];
  float (*red)[32][NV] = red_s[half];
  float (*hr)[SEG][32] = hr_s[half];
  float* part = need_norm ? st.lag_part + (size_t)seq * dm.max_new * (2 * dm.L) : nullptr;
  float* rpart = need_raw ? st.raw_part + (size_t)seq * dm.max_new * (2 * dm.L) : nullptr;
  int r = p0 % dm.lag;                   // position of the next token inside its chunk
  int parity = 0;

  for (int g0 = 0; g0 < n_new; g0 += kLagOffs) {
    const int gn = min(kLagOffs, n_new - g0);
    // one-token calls: every thread looks its row up itself (one broadcast
    // load per warp), so no shared table and none of its two barriers.  The
    // SEG == 1 instances run only in the decode-step kernel, whose calls
    // carry one token per sequence (it rejects n_new > 1), so the group holds
    // that one row.
    int64_t off1 = 0;
    if constexpr (SEG == 1 && EPIKV_TOKEN_OWN_OFFSET) {
      off1 = kv_row_offset(kv, layer, seq, nc0 + g0, dm.T);
    } else {
      __syncthreads();
      for (int t = tid; t < gn; t += nthr) soff[t] = kv_row_offset(kv, layer, seq, nc0 + g0 + t, dm.T);
      __syncthreads();
    }
    // rows are prefetched into L2 kLagPf segments ahead of their loads (whole
    // rows of H*d channels, one bulk prefetch each); the group's first ones here
    const uint32_t row_bytes = (uint32_t)hd * 2u;
    if constexpr (SEG > 1 && kLagPf > 0) {
      for (int t = tid; t < min(kLagPf * SEG, gn); t += nthr)
        if (soff[t] >= 0) prefetch_l2_bulk(kvbase + soff[t] * 2, row_bytes);
    }
    for (int i = 0; i < gn;) {
      const int seg = min(min(dm.lag - r, gn - i), SEG);
      const bool has_prev = p0 + g0 + i >= dm.lag;   // the segment's chunk is not chunk 0
      uint4 x[SEG];
      // FULL: every token of the segment is taken (the common case), so the
      // per-token conditions compile away; the arithmetic is the same
      auto body = [&](auto full_t, auto mom_t) {
        constexpr bool FULL = decltype(full_t)::value;
        constexpr bool MOM = decltype(mom_t)::value;  // has_prev && need_norm: the normalised moments
        int64_t offs[SEG];
        bool all_ok = active;
#pragma unroll
        for (int j = 0; j < SEG; ++j) {
          if constexpr (SEG == 1 && EPIKV_TOKEN_OWN_OFFSET) offs[j] = off1;
          else offs[j] = (FULL || j < seg) ? soff[i + j] : 0;
          all_ok &= offs[j] >= 0;
        }
        if (FULL && all_ok) {  // every row of the segment mapped: plain loads
#pragma unroll
          for (int j = 0; j < SEG; ++j) x[j] = ld_stream16(kvb_ch + offs[j] * 2);
        } else {
          bool bad = false;
#pragma unroll
          for (int j = 0; j < SEG; ++j) {
            const bool take = (FULL || j < seg) && active;
            bad |= take && offs[j] < 0;
            x[j] = ld_stream16_if(kvb_ch + offs[j] * 2, take && offs[j] >= 0);
          }
          if (bad) set_error(st.err, EPIKV_DEV_SLOT);
        }
        if constexpr (SEG > 1 && kLagPf > 0) {  // rows [i + kLagPf*SEG, + seg): every row once over the group
          const int t = i + kLagPf * SEG + tid;
          if (tid < seg && t < gn && soff[t] >= 0) prefetch_l2_bulk(kvbase + soff[t] * 2, row_bytes);
        }
        // two tokens at a time, so that rows' registers are free once used:
        // their raw variances, their normalised moments, then the running
        // range over both (the same min/max sequence as token by token)
        float v[NV];
        if (r == 0) {
          cmn = x[0];
          cmx = x[0];
        }
#pragma unroll
        for (int j0 = 0; j0 < SEG; j0 += 2) {
#pragma unroll
          for (int j = j0; j < j0 + 2 && j < SEG; ++j) {
            if (FULL || j < seg) {
              if (need_raw) {  // population variance of the stored vector over the head dimension
                float xf[8], s1 = 0.f;
                unpack8(x[j], xf);
#pragma unroll
                for (int e = 0; e < 8; ++e) s1 += xf[e];
                const float mean = group_sum(s1, LH) * inv_d;
                float s2 = 0.f;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                  const float dv = xf[e] - mean;
                  s2 = fmaf(dv, dv, s2);
                }
                const float var_raw = group_sum(s2, LH) * inv_d;
                if (q == 0 && active) hr[parity][j][h] = var_raw;
              }
              if constexpr (MOM) lag_moments(x[j], na, nc, v[2 * j], v[2 * j + 1]);
            } else if constexpr (MOM) {
              v[2 * j] = v[2 * j + 1] = 0.f;
            }
          }
          if (j0 + 1 < SEG && (FULL || j0 + 1 < seg)) {
            cmn = q_min(q_min(cmn, x[j0]), x[j0 + 1]);
            cmx = q_max(q_max(cmx, x[j0]), x[j0 + 1]);
          } else if (FULL || j0 < seg) {
            cmn = q_min(cmn, x[j0]);
            cmx = q_max(cmx, x[j0]);
          }
        }
        if constexpr (MOM) {
          transpose_sum<LH / 2, NV, NV>(v, tid & 31);
          if (active) {
            if constexpr (LH <= NV) {
#pragma unroll
              for (int k = 0; k < NV / LH; ++k) red[parity][h][k + (NV / LH) * q] = v[k];
            } else {
              if (q % (LH / NV) == 0) red[parity][h][q / (LH / NV)] = v[0];
            }
          }
        }
      };
      if (has_prev && need_norm) {
        if (seg == SEG) body(std::true_type{}, std::true_type{});
        else body(std::false_type{}, std::true_type{});
      } else {
        if (seg == SEG) body(std::true_type{}, std::false_type{});
        else body(std::false_type{}, std::false_type{});
      }
      __syncthreads();
      if (tid < seg) {
        if (need_norm) {
          float sum = 0.f;
          if (has_prev)
            for (int hh = 0; hh < dm.H; ++hh) {
              const float mean = red[parity][hh][2 * tid] * inv_d;
              sum += fmaxf(fmaf(-mean, mean, red[parity][hh][2 * tid + 1] * inv_d), 0.f);
            }
          part[(size_t)(g0 + i + tid) * (2 * dm.L) + stream] = sum;
        }
        if (need_raw) {
          float sum = 0.f;
          for (int hh = 0; hh < dm.H; ++hh) sum += hr[parity][tid][hh];
          rpart[(size_t)(g0 + i + tid) * (2 * dm.L) + stream] = sum;
        }
      }
      parity ^= 1;
      r += seg;
      if (r == dm.lag) {  // chunk complete: it becomes the previous chunk
        prev_affine(cmn, cmx, dm.lag_eps, na, nc);
        if (active && need_norm) {
          *reinterpret_cast<uint4*>(rng + 0 * hd + ch) = cmn;
          *reinterpret_cast<uint4*>(rng + 1 * hd + ch) = cmx;
        }
        r = 0;
      }
      i += seg;
    }
  }
  if (active && need_norm) {
    *reinterpret_cast<uint4*>(rng + 2 * hd + ch) = cmn;
    *reinterpret_cast<uint4*>(rng + 3 * hd + ch) = cmx;
  }
}

#ifndef EPIKV_LAG_MAXREG
#define EPIKV_LAG_MAXREG 72  // 7 CTAs of 128 threads per SM: 2,048 CTAs in two rounds (measured best; 64 spills)
#endif
#if EPIKV_LAG_MAXREG > 0
#define EPIKV_LAG_BOUNDS __maxnreg__(EPIKV_LAG_MAXREG)
#else
#define EPIKV_LAG_BOUNDS __launch_bounds__(256, EPIKV_LAG_MINB)
#endif
template <int LH, int KINDS>
__global__ void EPIKV_LAG_BOUNDS lagkv_partial_kernel(DevState st, Dims dm, KvDev kv,
                                                             const int32_t* __restrict__ seq_ids,
                                                             const int32_t* __restrict__ cu_new,
                                                             int max_new) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y;
  const int seq = seq_ids[b];
  const int n_new = cu_new[b + 1] - cu_new[b];
  if (seq < 0 || seq >= dm.S || n_new < 0 || n_new > max_new) {
    if (threadIdx.x == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  const int layer = blockIdx.x >> 1, kvk = blockIdx.x & 1;
  // the new rows' first slot: this layer's own length under per-layer budgets
  const int nc0 = dm.layer_budgets ? st.n_layer[seq * dm.L + layer] : st.n_cache[seq];
  if (nc0 + n_new > dm.T) {
    if (threadIdx.x == 0) set_error(st.err, EPIKV_DEV_CAPACITY);
    return;
  }
  lag_stream<LH, kLagSeg, false, KINDS>(st, dm, kv, seq, n_new, layer, kvk, nc0);
}

#ifndef EPIKV_FIN_TILE
#define EPIKV_FIN_TILE 16
#endif
constexpr int kFinTile = EPIKV_FIN_TILE;  // tokens per finalize CTA
constexpr int kFinThreads = 256;
constexpr int kMaxWindow = 1024;

// grid: (token tiles of 32, batch entries); block: 256 threads (warp per token).
template <int WPL>
__global__ void __launch_bounds__(kFinThreads) score_finalize_kernel(DevState st, Dims dm,
                                                                     const int32_t* __restrict__ seq_ids,
                                                                     const int32_t* __restrict__ cu_new,
                                                                     int max_new) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y;
  const int seq = seq_ids[b];
  const int n_new = cu_new[b + 1] - cu_new[b];
  if (seq < 0 || seq >= dm.S || n_new < 0 || n_new > max_new) {
    if (threadIdx.x == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nc0 = st.n_cache[seq];
  const int p0 = st.n_seen[seq];
  const bool fits = nc0 + n_new <= dm.T;
  if (!fits && tid == 0 && blockIdx.x == 0) set_error(st.err, EPIKV_DEV_CAPACITY);
  const int i_lo = blockIdx.x * kFinTile;
  const int i_hi = min(i_lo + kFinTile, n_new);
  const int Gm = dm.G - 1;
  const int nb = dm.nA + dm.nB;

  if (fits && i_lo < i_hi) {
    for (int i = i_lo + warp; i < i_hi; i += kFinThreads / 32) {
      const int pos = p0 + i;
      if (lane == 0) st.pos[(size_t)seq * dm.T + nc0 + i] = pos;
      if (lane == 0 && dm.layer_budgets)  // a new token is in every layer
        st.lmask[(size_t)seq * dm.T + nc0 + i] = dm.L == 64 ? ~0ull : (1ull << dm.L) - 1ull;
    }
    if (dm.kinds & kBandKinds) {
      // every g value the tile's windows reach, all band layers, one round of loads
      extern __shared__ float sg[];  // [nb][span]
      const int span = kFinTile + dm.z_window - 1;
      const int pos_base = p0 + i_lo - (dm.z_window - 1);  // position held by sg[band][0]
      const int pos_end = p0 + i_hi;
      for (int idx = tid; idx < nb * span; idx += kFinThreads) {
        const int band = idx / span;
        const int pos = pos_base + (idx - band * span);
        sg[idx] = (pos >= 1 && pos < pos_end) ? st.g_ring[((size_t)seq * nb + band) * dm.G + (pos & Gm)] : 0.f;
      }
      __syncthreads();
      // a lane per (token, band layer): lpt lanes per token, 32/lpt tokens per warp
      const int lpt = nb <= 16 ? 16 : 32;
      const int sub = lane / lpt, band = lane % lpt;
      for (int i0 = i_lo + warp * (32 / lpt); i0 < i_hi; i0 += kFinThreads / lpt) {
        const int i = i0 + sub;
        const int pos = p0 + i;
        const bool live = i < i_hi && pos >= 1 && band < nb;
        float za = 0.f, zb = 0.f, ma = 0.f, mb = 0.f;
        if (live) {
          const int n = min(dm.z_window, pos);
          const float* row = sg + band * span + (pos - pos_base);   // row[-k] = g at position pos - k
          if (dm.kinds & EPIKV_SCORE_BANDZ) {
            const float gnew = row[0];
            float dsum = 0.f;
            for (int k = 0; k < n; ++k) dsum += row[-k] - gnew;
            const float mean_d = dsum / (float)n;
            float dev = 0.f;
            for (int k = 0; k < n; ++k) {
              const float e = (row[-k] - gnew) - mean_d;
              dev = fmaf(e, e, dev);
            }
            const float sigma = sqrtf(dev / (float)n);
            const float z = -mean_d / (sigma + dm.z_eps);  // g(t) - mu = -(mean of g - g(t))
            if (band < dm.nA) za = z; else zb = z;
          }
          if (dm.kinds & EPIKV_SCORE_HSVAR) {  // rolling mean of g (Eq. 2)
            float sum = 0.f;
            for (int k = 0; k < n; ++k) sum += row[-k];
            const float gbar = sum / (float)n;
            if (band < dm.nA) ma = gbar; else mb = gbar;
          }
        }
        for (int o = lpt >> 1; o > 0; o >>= 1) {  // stays inside each token's lane group
          za += __shfl_xor_sync(0xffffffffu, za, o);
          zb += __shfl_xor_sync(0xffffffffu, zb, o);
          ma += __shfl_xor_sync(0xffffffffu, ma, o);
          mb += __shfl_xor_sync(0xffffffffu, mb, o);
        }
        if (band == 0 && i < i_hi) {
          const size_t slot = (size_t)seq * dm.T + nc0 + i;
          if (dm.kinds & EPIKV_SCORE_BANDZ)
            st.score[0][slot] = pos >= 1 ? za / (float)dm.nA - zb / (float)dm.nB : 0.f;
          if (dm.kinds & EPIKV_SCORE_HSVAR)
            st.score[2][slot] = pos >= 1 ? ma / (float)dm.nA - mb / (float)dm.nB : 0.f;
        }
      }
    }
    if (dm.kinds & kKvKinds) {
      __shared__ float su[kFinTile + kMaxWindow];
      const int w = dm.lag_window;
      const int lo = max(0, i_lo - (w - 1));
      const float inv_lh = 1.f / (float)(dm.L * dm.H);
      for (int qk = 0; qk < 4; ++qk) {
        const int kind = kv_kind(qk);
        if (!(dm.kinds & kind)) continue;
        // which partials: normalised or raw; all (layer, K|V) entries, keys only or values only
        const bool raw = kind & kRawKinds;
        const float* part = (raw ? st.raw_part : st.lag_part) + (size_t)seq * dm.max_new * (2 * dm.L);
        const int q0 = kind == EPIKV_SCORE_KVVAL ? 1 : 0;
        const int qs = kind == EPIKV_SCORE_LAGKV ? 1 : 2;
        float* ring = st.u_ring[qk] + (size_t)seq * dm.G;
        float* out = st.score[kind_index(kind)] + (size_t)seq * dm.T + nc0;
        __syncthreads();  // su is reused kind after kind
        for (int i = lo + tid; i < i_hi; i += kFinThreads) {
          const int pos = p0 + i;
          float u = 0.f;
          if (raw || pos >= dm.lag) {  // the normalised kinds have no value in chunk 0
            const float* pp = part + (size_t)i * (2 * dm.L);
            float s = 0.f;
            for (int q = q0; q < 2 * dm.L; q += qs) s += pp[q];
            u = s * inv_lh;
          }
          su[i - lo] = u;
        }
        __syncthreads();
        for (int i = i_lo + warp; i < i_hi; i += kFinThreads / 32) {
          const int pos = p0 + i;
          const int n = min(w, pos + 1);
          float acc = 0.f;
#pragma unroll
          for (int m = 0; m < WPL; ++m) {
            const int k = lane + 32 * m;
            if (k < n) acc += (i - k >= 0) ? su[i - k - lo] : ring[(pos - k) & Gm];
          }
          const float mean = warp_sum(acc) / (float)n;
          if (lane == 0) out[i] = mean;
        }
        for (int i = i_lo + tid; i < i_hi; i += kFinThreads) ring[(p0 + i) & Gm] = su[i - lo];
      }
    }
  }

  // The last CTA of this sequence commits its counters (no CTA waits).
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    const uint32_t done = atomicAdd(&st.ticket[seq], 1u);
    if (done == gridDim.x - 1) {
      __threadfence();
      if (fits) {
        // an eviction selected but not compacted before this update breaks the
        // call order; nothing is left pending for a later compaction either way
        if (st.first_changed[seq] < nc0) set_error(st.err, EPIKV_DEV_KEPT);
        st.first_changed[seq] = nc0 + n_new;
        st.n_cache[seq] = nc0 + n_new;
        st.n_seen[seq] = p0 + n_new;
        if (dm.layer_budgets)
          for (int l = 0; l < dm.L; ++l) {
            st.n_layer[seq * dm.L + l] += n_new;
            st.lfirst[seq * dm.L + l] = st.n_layer[seq * dm.L + l];
          }
        if ((dm.kinds & kBandKinds) && n_new > 0) st.hp_parity[seq] ^= 1;
        atomicAdd(&st.stats[0], (unsigned long long)n_new);
      }
      st.ticket[seq] = 0u;
    }
  }
}

// ---- one new token per sequence (a decode step)
#ifndef EPIKV_TOKEN_MINB
// token_kernel CTAs resident per SM: 5 caps registers at 48 (64 ragged
// sequences' decode step: 45.7 / 41.1 / 38.5 / 38.5 us at 3 / 4 / 5 / 6)
#define EPIKV_TOKEN_MINB 5
#endif

// One new token's g for one band layer (Eq. 1), from its row and the saved
// previous row (h_prev), exactly as bandz_g_kernel forms it (same per-thread
// vectors, fused multiply-adds, warp sums and fixed-order cross-warp sum);
// the row is saved as the next call's previous row.  Then, for the band
// kinds' scores (Eq. 3), this band's z of the new g against its window and
// the window's mean, with score_finalize_kernel's arithmetic and order (the
// shifted two-pass over g at positions pos, pos-1, ..., pos-n+1, one thread),
// stored per (sequence, band) for the last CTA to combine.  The window's
// earlier values are loaded with the rows into `win` (z_window floats of
// shared memory).  Every thread of a kGThreads block calls it.
template <int VPT>
__device__ __forceinline__ void band_token_g(const DevState& st, const Dims& dm, const BandRows& rows,
                                             int64_t row_stride, int band, int seq, int r0, int pos, int par,
                                             float* win) {
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nb = dm.nA + dm.nB;
  const int VR = dm.D >> 3;
  __shared__ float red[kGThreads / 32];
  const __nv_bfloat16* cur = rows.p[band] + (int64_t)r0 * row_stride;
  const __nv_bfloat16* prow = st.h_prev + ((size_t)(seq * 2 + par) * nb + band) * dm.D;
  __nv_bfloat16* hp_wr = st.h_prev + ((size_t)(seq * 2 + (par ^ 1)) * nb + band) * dm.D;
  float* ring = st.g_ring + ((size_t)seq * nb + band) * dm.G;
  const int n = pos >= 1 ? min(dm.z_window, pos) : 0;  // the new g's window, itself included
  uint4 c[VPT], p[VPT];
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int v = tid + k * kGThreads;
    c[k] = v < VR ? ld_stream16(cur + v * 8) : make_uint4(0, 0, 0, 0);
    p[k] = v < VR ? ld_stream16(prow + v * 8) : make_uint4(0, 0, 0, 0);
  }
  for (int k = 1 + tid; k < n; k += kGThreads) win[k] = __ldcg(ring + ((pos - k) & (dm.G - 1)));
  float acc = 0.f;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    float cf[8], pf[8];
    unpack8(c[k], cf);
    unpack8(p[k], pf);
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const float dlt = cf[e] - pf[e];
      acc = fmaf(dlt, dlt, acc);
    }
  }
  acc = warp_sum(acc);
  if (lane == 0) red[warp] = acc;
#pragma unroll
  for (int k = 0; k < VPT; ++k) {
    const int v = tid + k * kGThreads;
    if (v < VR) *reinterpret_cast<uint4*>(hp_wr + v * 8) = c[k];
  }
  __syncthreads();
  if (tid == 0) {
    float sum = 0.f;
#pragma unroll
    for (int w = 0; w < kGThreads / 32; ++w) sum += red[w];
    const float g = sqrtf(sum);
    if (pos >= 1) ring[pos & (dm.G - 1)] = g;
    if (n > 0) {
      win[0] = g;
      const float* row = win;  // row[k] = g at position pos - k
      float z = 0.f, gbar = 0.f;
      if (dm.kinds & EPIKV_SCORE_BANDZ) {
        const float gnew = row[0];
        float dsum = 0.f;
        for (int k = 0; k < n; ++k) dsum += row[k] - gnew;
        const float mean_d = dsum / (float)n;
        float dev = 0.f;
        for (int k = 0; k < n; ++k) {
          const float e = (row[k] - gnew) - mean_d;
          dev = fmaf(e, e, dev);
        }
        const float sigma = sqrtf(dev / (float)n);
        z = -mean_d / (sigma + dm.z_eps);
      }
      if (dm.kinds & EPIKV_SCORE_HSVAR) {
        float s = 0.f;
        for (int k = 0; k < n; ++k) s += row[k];
        gbar = s / (float)n;
      }
      st.ztok[(size_t)(seq * 2) * nb + band] = z;
      st.ztok[(size_t)(seq * 2 + 1) * nb + band] = gbar;
    }
  }
}

// The band kinds' scores of the new token at slot nc0: the per-band z and
// window means the band CTAs stored, combined exactly as
// score_finalize_kernel combines them (a lane per band, the same butterfly
// over the lanes).  One warp calls it.
__device__ __forceinline__ void band_token_combine(const DevState& st, const Dims& dm, int seq, int nc0, int pos) {
  const int lane = threadIdx.x & 31;
  const int nb = dm.nA + dm.nB;
  const int lpt = nb <= 16 ? 16 : 32;  // the lanes of one token, as in score_finalize_kernel
  const int bl = lane % lpt;
  const bool live = lane < lpt && pos >= 1 && bl < nb;
  float za = 0.f, zb = 0.f, ma = 0.f, mb = 0.f;
  if (live) {
    if (dm.kinds & EPIKV_SCORE_BANDZ) {
      const float z = __ldcg(st.ztok + (size_t)(seq * 2) * nb + bl);
      if (bl < dm.nA) za = z; else zb = z;
    }
    if (dm.kinds & EPIKV_SCORE_HSVAR) {
      const float gbar = __ldcg(st.ztok + (size_t)(seq * 2 + 1) * nb + bl);
      if (bl < dm.nA) ma = gbar; else mb = gbar;
    }
  }
  for (int o = lpt >> 1; o > 0; o >>= 1) {
    za += __shfl_xor_sync(0xffffffffu, za, o);
    zb += __shfl_xor_sync(0xffffffffu, zb, o);
    ma += __shfl_xor_sync(0xffffffffu, ma, o);
    mb += __shfl_xor_sync(0xffffffffu, mb, o);
  }
  if (lane == 0) {
    const size_t slot = (size_t)seq * dm.T + nc0;
    if (dm.kinds & EPIKV_SCORE_BANDZ) st.score[0][slot] = pos >= 1 ? za / (float)dm.nA - zb / (float)dm.nB : 0.f;
    if (dm.kinds & EPIKV_SCORE_HSVAR) st.score[2][slot] = pos >= 1 ? ma / (float)dm.nA - mb / (float)dm.nB : 0.f;
  }
}

// The K/V kinds' scores of the new token at slot nc0 (position pos), exactly
// as score_finalize_kernel forms them for a call's single token: u from the
// per-(layer, K|V) partials the stream CTAs wrote, summed in stream order by
// one thread (the warp first loads them into shared memory together, so the
// sum waits on one round of loads, not on 2L); its rolling mean over this u
// and the ring's earlier ones, a lane per window position in the same order,
// the same warp sum.  One warp calls it.
__device__ __forceinline__ void kv_token_scores(const DevState& st, const Dims& dm, int seq, int nc0, int pos) {
  const int lane = threadIdx.x & 31;
  __shared__ float pv[2 * 64];  // the host admits at most 64 layers
  const int Gm = dm.G - 1;
  const int w = dm.lag_window;
  const int n = min(w, pos + 1);
  const float inv_lh = 1.f / (float)(dm.L * dm.H);
  for (int qk = 0; qk < 4; ++qk) {
    const int kind = kv_kind(qk);
    if (!(dm.kinds & kind)) continue;
    const bool raw = kind & kRawKinds;
    const float* part = (raw ? st.raw_part : st.lag_part) + (size_t)seq * dm.max_new * (2 * dm.L);
    const int q0 = kind == EPIKV_SCORE_KVVAL ? 1 : 0;
    const int qs = kind == EPIKV_SCORE_LAGKV ? 1 : 2;
    float* ring = st.u_ring[qk] + (size_t)seq * dm.G;
    float u = 0.f;
    if (raw || pos >= dm.lag) {  // the normalised kinds have no value in chunk 0
      for (int q = lane; q < 2 * dm.L; q += 32) pv[q] = __ldcg(part + q);
      __syncwarp();
      if (lane == 0) {
        float s = 0.f;
        for (int q = q0; q < 2 * dm.L; q += qs) s += pv[q];
        u = s * inv_lh;
      }
      __syncwarp();  // pv is reused kind after kind
    }
    u = __shfl_sync(0xffffffffu, u, 0);
    float acc = 0.f;
    for (int k = lane; k < n; k += 32) acc += k == 0 ? u : __ldcg(ring + ((pos - k) & Gm));
    const float mean = warp_sum(acc) / (float)n;
    if (lane == 0) {
      st.score[kind_index(kind)][(size_t)seq * dm.T + nc0] = mean;
      ring[pos & Gm] = u;
    }
  }
}

// The decode step's commit of one sequence (as score_finalize_kernel's last
// CTA does it): the new slot's position, the counters, h_prev's parity.
// One thread.
__device__ __forceinline__ void token_commit(const DevState& st, const Dims& dm, int seq, int nc0, int pos) {
  const size_t slot = (size_t)seq * dm.T + nc0;
  st.pos[slot] = pos;
  if (dm.layer_budgets) {  // the new token is in every layer
    st.lmask[slot] = dm.L == 64 ? ~0ull : (1ull << dm.L) - 1ull;
    for (int l = 0; l < dm.L; ++l) {
      st.n_layer[seq * dm.L + l] += 1;
      st.lfirst[seq * dm.L + l] = st.n_layer[seq * dm.L + l];
    }
  }
  if (st.first_changed[seq] < nc0) set_error(st.err, EPIKV_DEV_KEPT);
  st.first_changed[seq] = nc0 + 1;
  st.n_cache[seq] = nc0 + 1;
  st.n_seen[seq] = pos + 1;
  if (dm.kinds & kBandKinds) st.hp_parity[seq] ^= 1;
  atomicAdd(&st.stats[0], 1ull);
  st.ticket[seq] = 0u;
}

// One new token per sequence with the band kinds only: g and the rolling
// z-score in one launch.  grid (band layers, batch entries), kGThreads
// threads: each CTA forms its band row's g and that band's z and window mean
// (band_token_g); the last CTA of a sequence (atomic ticket after a fence; no
// CTA waits) combines them into the scores (band_token_combine) and commits
// the sequence.  Results equal the two-kernel path bit for bit.
template <int VPT>
__global__ void __launch_bounds__(kGThreads) bandz_token_kernel(DevState st, Dims dm, BandRows rows,
                                                                 int64_t row_stride,
                                                                 const int32_t* __restrict__ seq_ids,
                                                                 const int32_t* __restrict__ cu_new) {
  pdl_wait();
  pdl_trigger();
  const int band = blockIdx.x, b = blockIdx.y;
  const int tid = threadIdx.x;
  const int seq = seq_ids[b];
  const int r0 = cu_new[b], n_new = cu_new[b + 1] - r0;
  if (seq < 0 || seq >= dm.S || n_new < 0 || n_new > 1 || cu_new[0] != 0) {
    if (tid == 0 && band == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  if (n_new == 0) return;
  const int nb = dm.nA + dm.nB;
  const int nc0 = st.n_cache[seq];
  const int pos = st.n_seen[seq];
  if (nc0 + 1 > dm.T) {
    if (tid == 0 && band == 0) set_error(st.err, EPIKV_DEV_CAPACITY);
    return;
  }
  __shared__ int s_last;
  extern __shared__ float win[];  // [z_window]: this band's window of g
  band_token_g<VPT>(st, dm, rows, row_stride, band, seq, r0, pos, st.hp_parity[seq], win);
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&st.ticket[seq], 1u) == (unsigned)(nb - 1);
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  if (tid < 32) band_token_combine(st, dm, seq, nc0, pos);
  if (tid == 32) token_commit(st, dm, seq, nc0, pos);  // meanwhile: they touch disjoint state
}

// One new token per sequence with a K/V kind (and any band kinds): the whole
// score update in one launch.  grid (band layers + L or 2L, batch entries),
// kGThreads threads: the first CTAs form the band rows' g, z and window means
// (band_token_g), the
// others the (layer, K|V) streams (lag_stream, the multi-token kernel's own
// code on a one-token call): a layer's K and V in the two halves of a CTA
// (`half`, when H*d/8 <= 128), else one stream per CTA; the last CTA of a
// sequence (ticket) forms every kind's score (band_token_combine,
// kv_token_scores) and commits.  Results equal the three-kernel path bit for
// bit.
template <int LH>
__global__ void __launch_bounds__(kGThreads, EPIKV_TOKEN_MINB) token_kernel(DevState st, Dims dm, BandRows rows, int64_t row_stride,
                                                           KvDev kv, const int32_t* __restrict__ seq_ids,
                                                           const int32_t* __restrict__ cu_new, int vpt, int half) {
  pdl_wait();
  pdl_trigger();
  const int b = blockIdx.y, tid = threadIdx.x;
  const int seq = seq_ids[b];
  const int r0 = cu_new[b], n_new = cu_new[b + 1] - r0;
  if (seq < 0 || seq >= dm.S || n_new < 0 || n_new > 1 || cu_new[0] != 0) {
    if (tid == 0 && blockIdx.x == 0) set_error(st.err, EPIKV_DEV_BATCH);
    return;
  }
  if (n_new == 0) return;
  const int nbc = (dm.kinds & kBandKinds) ? dm.nA + dm.nB : 0;  // band CTAs
  const int nc0 = st.n_cache[seq];
  const int pos = st.n_seen[seq];
  if (nc0 + 1 > dm.T) {
    if (tid == 0 && blockIdx.x == 0) set_error(st.err, EPIKV_DEV_CAPACITY);
    return;
  }
  __shared__ int s_last;
  extern __shared__ float win[];  // [z_window] (band CTAs): the band's window of g
  if ((int)blockIdx.x < nbc) {
    const int par = st.hp_parity[seq];
    if (vpt == 1) band_token_g<1>(st, dm, rows, row_stride, blockIdx.x, seq, r0, pos, par, win);
    else if (vpt == 2) band_token_g<2>(st, dm, rows, row_stride, blockIdx.x, seq, r0, pos, par, win);
    else band_token_g<4>(st, dm, rows, row_stride, blockIdx.x, seq, r0, pos, par, win);
  } else {
    const int sidx = blockIdx.x - nbc;
    const int layer = half ? sidx : sidx >> 1;
    // the new row's slot: this layer's own length under per-layer budgets
    const int lnc0 = dm.layer_budgets ? st.n_layer[seq * dm.L + layer] : nc0;
    if (half) lag_stream<LH, 1, true>(st, dm, kv, seq, 1, layer, threadIdx.x >> 7, lnc0);
    else lag_stream<LH, 1>(st, dm, kv, seq, 1, layer, sidx & 1, lnc0);
  }
  __syncthreads();
  if (tid == 0) {
    __threadfence();
    s_last = atomicAdd(&st.ticket[seq], 1u) == gridDim.x - 1;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // three warps at once, on disjoint state: the band scores (warp 0), the
  // K/V scores (warp 1) and the commit (warp 2)
  if (nbc && tid < 32) band_token_combine(st, dm, seq, nc0, pos);
  if (tid >= 32 && tid < 64) kv_token_scores(st, dm, seq, nc0, pos);
  if (tid == 64) token_commit(st, dm, seq, nc0, pos);
}

// ------------------------------------------------------------------ launchers
// dynamic shared memory of the finalize kernel: the band windows of a tile
static size_t finalize_smem(const Dims& dm) {
  if (!(dm.kinds & kBandKinds)) return 0;
  return (size_t)(dm.nA + dm.nB) * (kFinTile + dm.z_window - 1) * sizeof(float);
}

cudaError_t finalize_prepare() {
  const int mx = (int)((size_t)kMaxBand * (kFinTile + kMaxWindow - 1) * sizeof(float));
  const int wmx = (int)((size_t)kMaxBand * kMaxWindow * sizeof(float));
  cudaError_t e = cudaSuccess;
  auto allow = [&](auto kern, int bytes) {
    if (e == cudaSuccess) e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
  };
  allow(bandz_token_kernel<1>, wmx);
  allow(bandz_token_kernel<2>, wmx);
  allow(bandz_token_kernel<4>, wmx);
  allow(token_kernel<1>, wmx);
  allow(token_kernel<2>, wmx);
  allow(token_kernel<4>, wmx);
  allow(token_kernel<8>, wmx);
  allow(token_kernel<16>, wmx);
  allow(token_kernel<32>, wmx);
  allow(score_finalize_kernel<1>, mx);
  allow(score_finalize_kernel<2>, mx);
  allow(score_finalize_kernel<4>, mx);
  allow(score_finalize_kernel<8>, mx);
  allow(score_finalize_kernel<32>, mx);
  return e;
}

cudaError_t launch_score_update(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                                const int32_t* cu_new, int max_new, const epikv_hidden_view* hv,
                                const KvDev* kv, int num_sms, cudaStream_t stream, int* launches) {
  if (n_seq == 0 || max_new == 0) return cudaSuccess;
  const int nb = dm.nA + dm.nB;
  const bool band = dm.kinds & kBandKinds;
  BandRows rows;
  for (int i = 0; i < kMaxBand; ++i)
    rows.p[i] = band && i < nb ? static_cast<const __nv_bfloat16*>(hv->band_rows[i]) : nullptr;
  const int64_t rs = band ? hv->row_stride : 0;
  const int vr = dm.D / 8;
  const int vpt = vr <= kGThreads ? 1 : vr <= 2 * kGThreads ? 2 : 4;  // band row vectors per thread
  if (max_new == 1 && !(dm.kinds & kKvKinds)) {  // a decode step of the band kinds: one fused launch
    const dim3 grid(nb, n_seq);
    const size_t wsm = (size_t)dm.z_window * sizeof(float);  // a band CTA's window of g
    auto go = [&](auto kern) { pdl_launch(kern, grid, kGThreads, wsm, stream, st, dm, rows, rs, seq_ids, cu_new); };
    if (vpt == 1) go(bandz_token_kernel<1>);
    else if (vpt == 2) go(bandz_token_kernel<2>);
    else go(bandz_token_kernel<4>);
    ++*launches;
    return cudaGetLastError();
  }
  if (max_new == 1 && dm.L <= 64) {  // a decode step with a K/V kind: one fused launch
    const int half = dm.H * dm.d / 8 <= 128;  // a layer's K and V streams share a CTA
    const dim3 grid((band ? nb : 0) + (half ? dm.L : 2 * dm.L), n_seq);
    const size_t wsm = band ? (size_t)dm.z_window * sizeof(float) : 0;
    auto go = [&](auto kern) {
      pdl_launch(kern, grid, kGThreads, wsm, stream, st, dm, rows, rs, *kv, seq_ids, cu_new, vpt, half);
    };
    switch (dm.d / 8) {
      case 1: go(token_kernel<1>); break;
      case 2: go(token_kernel<2>); break;
      case 4: go(token_kernel<4>); break;
      case 8: go(token_kernel<8>); break;
      case 16: go(token_kernel<16>); break;
      default: go(token_kernel<32>); break;
    }
    ++*launches;
    return cudaGetLastError();
  }
  if (band) {
    // persistent: as many CTAs as are resident, never more than rows
    static int resident[3] = {0, 0, 0};
    const int vi = vpt == 1 ? 0 : vpt == 2 ? 1 : 2;
    if (!resident[vi]) {
      int per_sm = 1;
      if (vi == 0) cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, bandz_g_kernel<1>, kGThreads, 0);
      if (vi == 1) cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, bandz_g_kernel<2>, kGThreads, 0);
      if (vi == 2) cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, bandz_g_kernel<4>, kGThreads, 0);
      resident[vi] = (per_sm > 0 ? per_sm : 1) * num_sms;
    }
    const int64_t rows_bound = (int64_t)nb * n_seq * max_new;
    const int grid = (int)(rows_bound < resident[vi] ? rows_bound : resident[vi]);
    auto go = [&](auto kern) {
      pdl_launch(kern, grid, kGThreads, 0, stream, st, dm, rows, rs, seq_ids, cu_new, n_seq, max_new);
    };
    if (vi == 0) go(bandz_g_kernel<1>);
    else if (vi == 1) go(bandz_g_kernel<2>);
    else go(bandz_g_kernel<4>);
    ++*launches;
  }
  if (dm.kinds & kKvKinds) {
    const dim3 grid(2 * dm.L, n_seq);
    const int threads = max(32, (dm.H * dm.d / 8 + 31) / 32 * 32);
    auto go = [&](auto kern) { pdl_launch(kern, grid, threads, 0, stream, st, dm, *kv, seq_ids, cu_new, max_new); };
    auto lanes = [&](auto kinds_t) {
      constexpr int KS = decltype(kinds_t)::value;
      switch (dm.d / 8) {
        case 1: go(lagkv_partial_kernel<1, KS>); break;
        case 2: go(lagkv_partial_kernel<2, KS>); break;
        case 4: go(lagkv_partial_kernel<4, KS>); break;
        case 8: go(lagkv_partial_kernel<8, KS>); break;
        case 16: go(lagkv_partial_kernel<16, KS>); break;
        default: go(lagkv_partial_kernel<32, KS>); break;
      }
    };
    const int ks = ((dm.kinds & kNormKinds) ? 1 : 0) | ((dm.kinds & kRawKinds) ? 2 : 0);
    if (ks == 1) lanes(std::integral_constant<int, 1>{});
    else if (ks == 2) lanes(std::integral_constant<int, 2>{});
    else lanes(std::integral_constant<int, 0>{});   // both: the runtime flags (fewer spills than both fixed)
    ++*launches;
  }
  {
    const dim3 grid((max_new + kFinTile - 1) / kFinTile, n_seq);
    const int wmax = max(band ? dm.z_window : 1, (dm.kinds & kKvKinds) ? dm.lag_window : 1);
    const int wpl = (wmax + 31) / 32;
    const size_t smem = finalize_smem(dm);
    auto go = [&](auto kern) { pdl_launch(kern, grid, kFinThreads, smem, stream, st, dm, seq_ids, cu_new, max_new); };
    if (wpl <= 1) go(score_finalize_kernel<1>);
    else if (wpl <= 2) go(score_finalize_kernel<2>);
    else if (wpl <= 4) go(score_finalize_kernel<4>);
    else if (wpl <= 8) go(score_finalize_kernel<8>);
    else go(score_finalize_kernel<32>);
    ++*launches;
  }
  return cudaGetLastError();
}

}  // namespace epikv
