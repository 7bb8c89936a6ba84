// epikv_lagkv_score_noalloc: Lag-KV scores of a sequence's first n tokens in
// one call, for callers that cannot allocate device memory at all.
//
// Who needs it: a plugin running inside a host application whose own memory
// pool owns the whole device and refuses outside allocations, an embedded
// caller with no allocator bound to the GPU, or a latency-critical loop where
// a cudaMalloc (which can synchronise the device) is not acceptable.  Such a
// caller cannot create the workspace epikv_init needs, so this entry point
// keeps its working memory in a fixed array compiled into the library.
//
// The scratch is `g_noalloc_scratch`, a file-scope static device array of
// kNoallocScratchFloats floats (2 MiB).  Every GPU that loads the library
// holds it until the process exits.  In host code that name is only a host
// stand-in, not a device address: the first call in each CUDA context (with
// that context's device current) looks the real address up with
// cudaGetSymbolAddress and remembers it under the context's unique id, so a
// context that is torn down and created again (cudaDeviceReset) gets a fresh
// lookup instead of a stale address; that set-up is why the first call in a
// context should come before any stream capture.  The array is shared by
// every call and keeps the previous call's contents; every entry a call reads
// is written by the same call first, so nothing needs clearing, but two calls
// that overlap on the GPU (different streams, no ordering between them) race
// on it.
//
// Slots the view does not map (a negative or out-of-range block-table entry)
// are read as zero rows: this entry point has no error word, so such input
// is not reported.
//
// The kernels are variants of the Lag-KV partial and finalize kernels of the
// context path, for a sequence whose slots 0..n-1 hold positions 0..n-1.  They
// take each head's variance in two passes (mean, then squared deviations),
// where the context path uses shifted moments in one pass, so the scores agree
// with epikv_score_update's to fp32 rounding, not bit for bit.
#include <cuda.h>

#include <mutex>

#include "common.cuh"

namespace {

constexpr size_t kNoallocScratchFloats = size_t(1) << 19;  // 2 MiB: n * 2 * num_layers floats
constexpr int kMaxContexts = 64;  // contexts whose scratch address is remembered
constexpr int kBatch = 16;
constexpr int kTile = 32;
constexpr int kThreads = 256;

}  // namespace

static __device__ __align__(256) float g_noalloc_scratch[kNoallocScratchFloats];

namespace {

using epikv::KvDev;

// grid: 2L (layer, K|V); block: max(32, H*d/8) threads, d/8 lanes per head.
template <int LH>
__global__ void __launch_bounds__(256) noalloc_partial_kernel(KvDev kv, int seq, int n, int L, int H, int d,
                                                              int lag, float lag_eps, float* part) {
  const int layer = blockIdx.x >> 1, kvk = blockIdx.x & 1;
  const int tid = threadIdx.x;
  const int h = tid / LH, q = tid % LH;
  const bool active = h < H;
  const int ch = h * d + q * 8;
  float pmn[8], pmx[8], cmn[8], cmx[8], inv[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    pmn[e] = pmx[e] = cmn[e] = cmx[e] = 0.f;
    inv[e] = 1.f / (pmx[e] - pmn[e] + lag_eps);
  }
  const float inv_d = 1.f / (float)d;
  const char* base = kv.base[kvk];
  __shared__ float hv[kBatch][32];
  for (int i0 = 0; i0 < n; i0 += kBatch) {
    const int nbt = min(kBatch, n - i0);
    uint4 x[kBatch];
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      x[j] = make_uint4(0, 0, 0, 0);
      if (j < nbt && active) {
        const int64_t off = epikv::kv_row_offset(kv, layer, seq, i0 + j, n);
        if (off >= 0) x[j] = epikv::ld_stream16(base + (off + ch) * 2);
      }
    }
#pragma unroll
    for (int j = 0; j < kBatch; ++j) {
      if (j < nbt) {
        const int pos = i0 + j;
        const int c = pos / lag;
        const int r = pos - c * lag;
        float xf[8];
        epikv::unpack8(x[j], xf);
        float var = 0.f;
        if (c >= 1) {
          float xn[8], s = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            xn[e] = (xf[e] - pmn[e]) * inv[e];
            s += xn[e];
          }
          const float mean = epikv::group_sum(s, LH) * inv_d;
          float ss = 0.f;
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            const float dv = xn[e] - mean;
            ss = fmaf(dv, dv, ss);
          }
          var = epikv::group_sum(ss, LH) * inv_d;
        }
        if (q == 0 && active) hv[j][h] = var;
        if (r == 0) {
#pragma unroll
          for (int e = 0; e < 8; ++e) cmn[e] = cmx[e] = xf[e];
        } else {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            cmn[e] = fminf(cmn[e], xf[e]);
            cmx[e] = fmaxf(cmx[e], xf[e]);
          }
        }
        if (r == lag - 1) {
#pragma unroll
          for (int e = 0; e < 8; ++e) {
            pmn[e] = cmn[e];
            pmx[e] = cmx[e];
            inv[e] = 1.f / (pmx[e] - pmn[e] + lag_eps);
          }
        }
      }
    }
    __syncthreads();
    if (tid < nbt) {
      float s = 0.f;
      for (int hh = 0; hh < H; ++hh) s += hv[tid][hh];
      part[(size_t)(i0 + tid) * (2 * L) + blockIdx.x] = s;
    }
    __syncthreads();
  }
}

// grid: token tiles of 32; block: 256 threads, a warp per token.
template <int WPL>
__global__ void __launch_bounds__(kThreads) noalloc_finalize_kernel(const float* part, int n, int L, int H, int lag,
                                                                    int w, float* out) {
  __shared__ float su[kTile + 1024];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int i_lo = blockIdx.x * kTile, i_hi = min(i_lo + kTile, n);
  const int lo = max(0, i_lo - (w - 1));
  const float inv_lh = 1.f / (float)(L * H);
  for (int i = lo + tid; i < i_hi; i += kThreads) {
    float u = 0.f;
    if (i >= lag) {
      const float* pp = part + (size_t)i * (2 * L);
      float s = 0.f;
      for (int q = 0; q < 2 * L; ++q) s += pp[q];
      u = s * inv_lh;
    }
    su[i - lo] = u;
  }
  __syncthreads();
  for (int i = i_lo + warp; i < i_hi; i += kThreads / 32) {
    const int cnt = min(w, i + 1);
    float acc = 0.f;
#pragma unroll
    for (int m = 0; m < WPL; ++m) {
      const int k = lane + 32 * m;
      if (k < cnt) acc += su[i - k - lo];
    }
    const float mean = epikv::warp_sum(acc) / (float)cnt;
    if (lane == 0) out[i] = mean;
  }
}

// The current context's unique id (driver entry points fetched through the
// runtime, so the library needs no link-time dependency on the driver).
typedef CUresult (*CtxGetCurrentFn)(CUcontext*);
typedef CUresult (*CtxGetIdFn)(CUcontext, unsigned long long*);

std::mutex g_mu;
CtxGetCurrentFn g_ctx_current = nullptr;
CtxGetIdFn g_ctx_id = nullptr;
struct ScratchEntry {
  unsigned long long ctx_id;
  float* ptr;
};
ScratchEntry g_scratch[kMaxContexts] = {};
int g_scratch_next = 0;

cudaError_t current_context_id(unsigned long long* id) {
  if (!g_ctx_current || !g_ctx_id) {
    void* f1 = nullptr;
    void* f2 = nullptr;
    cudaDriverEntryPointQueryResult q1, q2;
    cudaError_t e = cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 12000, cudaEnableDefault, &q1);
    if (e == cudaSuccess) e = cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2);
    if (e != cudaSuccess) return e;
    if (q1 != cudaDriverEntryPointSuccess || q2 != cudaDriverEntryPointSuccess || !f1 || !f2)
      return cudaErrorNotSupported;
    g_ctx_current = reinterpret_cast<CtxGetCurrentFn>(f1);
    g_ctx_id = reinterpret_cast<CtxGetIdFn>(f2);
  }
  CUcontext ctx = nullptr;
  if (g_ctx_current(&ctx) != CUDA_SUCCESS || !ctx) return cudaErrorDeviceUninitialized;
  return g_ctx_id(ctx, id) == CUDA_SUCCESS ? cudaSuccess : cudaErrorContextIsDestroyed;
}

// Device address of the scratch array in the current context: looked up once
// per context, then taken from the table.
cudaError_t scratch_address(float** out) {
  std::lock_guard<std::mutex> lock(g_mu);
  unsigned long long id = 0;
  if (current_context_id(&id) == cudaSuccess)
    for (const ScratchEntry& s : g_scratch)
      if (s.ptr && s.ctx_id == id) {
        *out = s.ptr;
        return cudaSuccess;
      }
  // first call in this context (this also makes the device's primary context
  // current if no context was yet)
  void* p = nullptr;
  cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  e = current_context_id(&id);
  if (e != cudaSuccess) return e;
  g_scratch[g_scratch_next] = ScratchEntry{id, static_cast<float*>(p)};
  g_scratch_next = (g_scratch_next + 1) % kMaxContexts;
  *out = static_cast<float*>(p);
  return cudaSuccess;
}

bool view_ok(const epikv_kv_view* kv, int H, int d, KvDev* out) {
  if (!kv || !kv->k || !kv->v || ((uintptr_t)kv->k & 15u) || ((uintptr_t)kv->v & 15u)) return false;
  if (kv->stride_token < (int64_t)H * d || kv->stride_token % 8 || kv->stride_layer < 0 || kv->stride_layer % 8)
    return false;
  *out = KvDev{};
  out->base[0] = static_cast<char*>(kv->k);
  out->base[1] = static_cast<char*>(kv->v);
  out->layout = kv->layout;
  out->stride_layer = kv->stride_layer;
  out->stride_token = kv->stride_token;
  if (kv->layout == EPIKV_LAYOUT_CONTIGUOUS) {
    if (kv->stride_seq < 0 || kv->stride_seq % 8) return false;
    out->stride_seq = kv->stride_seq;
    return true;
  }
  if (kv->layout != EPIKV_LAYOUT_PAGED || !kv->block_table || kv->block_size < 1 || kv->max_blocks_per_seq < 1 ||
      kv->num_blocks < 1 || kv->stride_block < 0 || kv->stride_block % 8 || kv->stride_table_layer < 0)
    return false;
  out->stride_block = kv->stride_block;
  out->table_stride_layer = kv->stride_table_layer;
  out->block_table = kv->block_table;
  out->max_blocks = kv->max_blocks_per_seq;
  out->block_size = kv->block_size;
  out->num_blocks = kv->num_blocks;
  return true;
}

}  // namespace

extern "C" epikv_status epikv_lagkv_score_noalloc(const epikv_kv_view* kv, int32_t seq, int32_t n,
                                                  int32_t num_layers, int32_t num_kv_heads, int32_t head_dim,
                                                  int32_t lag, float lag_eps, int32_t window, float* d_scores,
                                                  cudaStream_t stream) {
  const int L = num_layers, H = num_kv_heads, d = head_dim;
  if (n < 1 || seq < 0 || L < 1 || H < 1 || H > 32 || d < 8 || d > 256 || (d & (d - 1)) || H * d / 8 > 256)
    return EPIKV_EINVAL;
  if (lag < 1 || window < 1 || window > 1024 || !(lag_eps >= 0.f) || !d_scores || ((uintptr_t)d_scores & 3u))
    return EPIKV_EINVAL;
  if ((size_t)n * 2 * (size_t)L > kNoallocScratchFloats) return EPIKV_EINVAL;  // beyond the fixed scratch
  KvDev kd;
  if (!view_ok(kv, H, d, &kd)) return EPIKV_EINVAL;
  // an error left by earlier, unrelated work stays with its owner: report it
  // without launching and without clearing it
  if (cudaPeekAtLastError() != cudaSuccess) return EPIKV_ECUDA;
  float* part = nullptr;
  if (scratch_address(&part) != cudaSuccess) return EPIKV_ECUDA;

  const int threads = (H * d / 8 + 31) / 32 * 32 < 32 ? 32 : (H * d / 8 + 31) / 32 * 32;
  const dim3 g1(2 * L);
  switch (d / 8) {
    case 1: noalloc_partial_kernel<1><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
    case 2: noalloc_partial_kernel<2><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
    case 4: noalloc_partial_kernel<4><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
    case 8: noalloc_partial_kernel<8><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
    case 16: noalloc_partial_kernel<16><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
    default: noalloc_partial_kernel<32><<<g1, threads, 0, stream>>>(kd, seq, n, L, H, d, lag, lag_eps, part); break;
  }
  const dim3 g2((n + kTile - 1) / kTile);
  const int wpl = (window + 31) / 32;
  if (wpl <= 1)
    noalloc_finalize_kernel<1><<<g2, kThreads, 0, stream>>>(part, n, L, H, lag, window, d_scores);
  else if (wpl <= 2)
    noalloc_finalize_kernel<2><<<g2, kThreads, 0, stream>>>(part, n, L, H, lag, window, d_scores);
  else if (wpl <= 4)
    noalloc_finalize_kernel<4><<<g2, kThreads, 0, stream>>>(part, n, L, H, lag, window, d_scores);
  else if (wpl <= 8)
    noalloc_finalize_kernel<8><<<g2, kThreads, 0, stream>>>(part, n, L, H, lag, window, d_scores);
  else
    noalloc_finalize_kernel<32><<<g2, kThreads, 0, stream>>>(part, n, L, H, lag, window, d_scores);
  // no error was pending before the launches, so any error now is theirs
  return cudaGetLastError() == cudaSuccess ? EPIKV_OK : EPIKV_ECUDA;
}
