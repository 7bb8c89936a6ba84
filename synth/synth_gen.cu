// Device twin of synth/gen.py: writes the same bf16 bytes as the numpy
// generator, for hidden-state rows and for K/V rows placed into a cache view
// (contiguous or paged).  It holds none of the eviction method's arithmetic.
// Every float operation is an explicitly rounded intrinsic so no FMA
// contraction can change a bit relative to the numpy side.
#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

namespace {

constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;
constexpr uint64_t kMul1 = 0xBF58476D1CE4E5B9ull;
constexpr uint64_t kMul2 = 0x94D049BB133111EBull;
constexpr uint64_t S_HIDDEN = 1, S_SEGMENT = 2, S_SPIKE = 3, S_KEY = 4, S_VALUE = 5;

__device__ __forceinline__ uint64_t mix64(uint64_t x) {
  uint64_t z = x + kGamma;
  z = (z ^ (z >> 30)) * kMul1;
  z = (z ^ (z >> 27)) * kMul2;
  return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t row_key(uint64_t stream, uint64_t seed, uint64_t seq, uint64_t layer,
                                             uint64_t head, uint64_t pos) {
  uint64_t k = mix64(mix64(seed) ^ stream);
  k = mix64(k ^ seq);
  k = mix64(k ^ ((layer << 16) | head));
  return mix64(k ^ pos);
}

__device__ __forceinline__ float normal16(uint64_t e) {
  const int s = (int)(e & 0xFFFF) + (int)((e >> 16) & 0xFFFF) + (int)((e >> 32) & 0xFFFF) + (int)(e >> 48);
  return (float)(s - 131070);  // exact
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  const uint32_t lo = __bfloat16_as_ushort(__float2bfloat16_rn(a));
  const uint32_t hi = __bfloat16_as_ushort(__float2bfloat16_rn(b));
  return lo | (hi << 16);
}

__global__ void hidden_kernel(uint64_t seed, int seq, int layer, int pos0, int n, int D, float scale, float drift,
                              float seg_amp, float inv_sd, const float* __restrict__ mean,
                              const int32_t* __restrict__ seg, uint16_t* __restrict__ out, int64_t row_stride) {
  const int t = blockIdx.x;
  if (t >= n) return;
  const int pos = pos0 + t;
  const uint64_t key = row_key(S_HIDDEN, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)pos);
  const float tf = __fmul_rn((float)pos, 1.52587890625e-05f);  // exact: pos * 2^-16
  const float c = __fmul_rn(__fmul_rn(scale, __fadd_rn(1.0f, __fmul_rn(drift, tf))), inv_sd);
  const bool has_seg = seg_amp != 0.0f;
  const float bamp = __fmul_rn(seg_amp, inv_sd);
  const uint64_t skey = has_seg ? row_key(S_SEGMENT, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)seg[pos]) : 0;
  uint16_t* row = out + (int64_t)t * row_stride;
  for (int v = threadIdx.x; v < D / 8; v += blockDim.x) {
    float f[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int j = v * 8 + e;
      float x = __fmul_rn(normal16(mix64(key + (uint64_t)j)), c);
      if (has_seg) x = __fadd_rn(x, __fmul_rn(normal16(mix64(skey + (uint64_t)j)), bamp));
      f[e] = __fadd_rn(x, mean[j]);
    }
    uint4 q;
    q.x = pack2(f[0], f[1]);
    q.y = pack2(f[2], f[3]);
    q.z = pack2(f[4], f[5]);
    q.w = pack2(f[6], f[7]);
    *reinterpret_cast<uint4*>(row + v * 8) = q;
  }
}

struct View {
  char* base[2];
  int layout;  // 0 contiguous, 1 paged
  int64_t stride_layer, stride_seq, stride_block, stride_token;
  const int32_t* block_table;
  int max_blocks, block_size;
};

// grid (n tokens, L layers, 2 kinds); block = H*d/8 threads (8 channels each)
__global__ void kv_kernel(uint64_t seed, int seq, int pos0, int n, int slot0, int L, int H, int d,
                          int spike_per_10k, const float* __restrict__ kv_scale, const float* __restrict__ kv_off,
                          View vw) {
  const int t = blockIdx.x, layer = blockIdx.y, kind = blockIdx.z;
  const int lpt = d / 8;
  const int h = threadIdx.x / lpt, j0 = (threadIdx.x % lpt) * 8;
  if (t >= n || h >= H) return;
  const int pos = pos0 + t, slot = slot0 + t;
  const uint64_t sp = row_key(S_SPIKE, seed, (uint64_t)seq, 0, 0, (uint64_t)pos);
  const bool spike = pos >= 1 && (sp % 10000ull) < (uint64_t)spike_per_10k;
  const float cs = __fmul_rn(kv_scale[(kind * L + layer) * H + h], spike ? 4.0f : 1.0f);
  const uint64_t key = row_key(kind == 0 ? S_KEY : S_VALUE, seed, (uint64_t)seq, (uint64_t)layer, (uint64_t)h,
                               (uint64_t)pos);
  const float* off = kv_off + ((int64_t)(kind * L + layer) * H + h) * d;
  float f[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int j = j0 + e;
    f[e] = __fadd_rn(__fmul_rn(normal16(mix64(key + (uint64_t)j)), cs), off[j]);
  }
  int64_t row;
  if (vw.layout == 0) {
    row = (int64_t)layer * vw.stride_layer + (int64_t)seq * vw.stride_seq + (int64_t)slot * vw.stride_token;
  } else {
    const int blk = vw.block_table[(int64_t)seq * vw.max_blocks + slot / vw.block_size];
    row = (int64_t)layer * vw.stride_layer + (int64_t)blk * vw.stride_block +
          (int64_t)(slot % vw.block_size) * vw.stride_token;
  }
  uint4 q;
  q.x = pack2(f[0], f[1]);
  q.y = pack2(f[2], f[3]);
  q.z = pack2(f[4], f[5]);
  q.w = pack2(f[6], f[7]);
  *reinterpret_cast<uint4*>(vw.base[kind] + (row + h * d + j0) * 2) = q;
}

// Batched rows: row i is (seqs[i], pos[i]); seg is [n_seq][seg_stride].
__global__ void hidden_batch_kernel(uint64_t seed, int layer, int n, const int32_t* __restrict__ seqs,
                                    const int32_t* __restrict__ poss, int D, float scale, float drift,
                                    float seg_amp, float inv_sd, const float* __restrict__ mean,
                                    const int32_t* __restrict__ seg, int64_t seg_stride, uint16_t* __restrict__ out,
                                    int64_t row_stride) {
  const int t = blockIdx.x;
  if (t >= n) return;
  const int seq = seqs[t], pos = poss[t];
  const uint64_t key = row_key(S_HIDDEN, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)pos);
  const float tf = __fmul_rn((float)pos, 1.52587890625e-05f);
  const float c = __fmul_rn(__fmul_rn(scale, __fadd_rn(1.0f, __fmul_rn(drift, tf))), inv_sd);
  const bool has_seg = seg_amp != 0.0f;
  const float bamp = __fmul_rn(seg_amp, inv_sd);
  const uint64_t skey =
      has_seg ? row_key(S_SEGMENT, seed, (uint64_t)seq, (uint64_t)layer, 0, (uint64_t)seg[seq * seg_stride + pos]) : 0;
  uint16_t* row = out + (int64_t)t * row_stride;
  for (int v = threadIdx.x; v < D / 8; v += blockDim.x) {
    float f[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const int j = v * 8 + e;
      float x = __fmul_rn(normal16(mix64(key + (uint64_t)j)), c);
      if (has_seg) x = __fadd_rn(x, __fmul_rn(normal16(mix64(skey + (uint64_t)j)), bamp));
      f[e] = __fadd_rn(x, mean[j]);
    }
    uint4 q;
    q.x = pack2(f[0], f[1]);
    q.y = pack2(f[2], f[3]);
    q.z = pack2(f[4], f[5]);
    q.w = pack2(f[6], f[7]);
    *reinterpret_cast<uint4*>(row + v * 8) = q;
  }
}

// grid (n rows, L, 2); row i = (seqs[i], pos[i]) written to slot slots[i].
__global__ void kv_batch_kernel(uint64_t seed, int n, const int32_t* __restrict__ seqs,
                                const int32_t* __restrict__ poss, const int32_t* __restrict__ slots, int L, int H,
                                int d, int spike_per_10k, const float* __restrict__ kv_scale,
                                const float* __restrict__ kv_off, View vw) {
  const int t = blockIdx.x, layer = blockIdx.y, kind = blockIdx.z;
  const int lpt = d / 8;
  const int h = threadIdx.x / lpt, j0 = (threadIdx.x % lpt) * 8;
  if (t >= n || h >= H) return;
  const int seq = seqs[t], pos = poss[t], slot = slots[t];
  const uint64_t sp = row_key(S_SPIKE, seed, (uint64_t)seq, 0, 0, (uint64_t)pos);
  const bool spike = pos >= 1 && (sp % 10000ull) < (uint64_t)spike_per_10k;
  const float cs = __fmul_rn(kv_scale[(kind * L + layer) * H + h], spike ? 4.0f : 1.0f);
  const uint64_t key = row_key(kind == 0 ? S_KEY : S_VALUE, seed, (uint64_t)seq, (uint64_t)layer, (uint64_t)h,
                               (uint64_t)pos);
  const float* off = kv_off + ((int64_t)(kind * L + layer) * H + h) * d;
  float f[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int j = j0 + e;
    f[e] = __fadd_rn(__fmul_rn(normal16(mix64(key + (uint64_t)j)), cs), off[j]);
  }
  int64_t row;
  if (vw.layout == 0) {
    row = (int64_t)layer * vw.stride_layer + (int64_t)seq * vw.stride_seq + (int64_t)slot * vw.stride_token;
  } else {
    const int blk = vw.block_table[(int64_t)seq * vw.max_blocks + slot / vw.block_size];
    row = (int64_t)layer * vw.stride_layer + (int64_t)blk * vw.stride_block +
          (int64_t)(slot % vw.block_size) * vw.stride_token;
  }
  uint4 q;
  q.x = pack2(f[0], f[1]);
  q.y = pack2(f[2], f[3]);
  q.z = pack2(f[4], f[5]);
  q.w = pack2(f[6], f[7]);
  *reinterpret_cast<uint4*>(vw.base[kind] + (row + h * d + j0) * 2) = q;
}

// Delivery of host-resident inputs (and read-back of results): row r (of
// gridDim.y) of `width16` 16-byte vectors, copied by the SMs through unified
// addressing (no copy engine), from pinned host memory to device memory or
// from device memory to pinned host memory.
__global__ void upload_kernel(char* __restrict__ dst, size_t dpitch, const char* __restrict__ src, size_t spitch,
                              size_t width16) {
  const size_t r = blockIdx.y;
  for (size_t c = blockIdx.x * (size_t)blockDim.x + threadIdx.x; c < width16; c += (size_t)gridDim.x * blockDim.x)
    *reinterpret_cast<uint4*>(dst + r * dpitch + c * 16) = *reinterpret_cast<const uint4*>(src + r * spitch + c * 16);
}

}  // namespace

extern "C" {

// `height` rows of `width` bytes from pinned host memory (rows `spitch` apart)
// to device memory (rows `dpitch` apart), or the other way, copied by about
// `ctas` CTAs of SM loads and stores over the host link: the input delivery
// and result read-back of the end-to-end measurement.  Pointers, pitches and
// width are 16-byte multiples.
int synth_upload_2d(void* dst, size_t dpitch, const void* src, size_t spitch, size_t width, size_t height, int ctas,
                    cudaStream_t stream) {
  if (!dst || !src || ctas < 1 || (width & 15) || (dpitch & 15) || (spitch & 15) || ((uintptr_t)dst & 15) ||
      ((uintptr_t)src & 15) || width > dpitch || width > spitch || height > 65535)
    return 1;
  if (width == 0 || height == 0) return 0;
  const int gx = ctas / (int)height > 0 ? ctas / (int)height : 1;
  upload_kernel<<<dim3(gx, (unsigned)height), 512, 0, stream>>>(static_cast<char*>(dst), dpitch,
                                                                static_cast<const char*>(src), spitch, width / 16);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// Rows [n][D] of one hidden layer for positions pos0..pos0+n-1 of one sequence.
int synth_hidden(uint64_t seed, int seq, int layer, int pos0, int n, int D, float scale, float drift, float seg_amp,
                 float inv_sd, const float* d_mean, const int32_t* d_seg, void* d_out, int64_t row_stride,
                 cudaStream_t stream) {
  if (n <= 0) return 0;
  if (D % 8 || !d_mean || !d_out || (seg_amp != 0.0f && !d_seg)) return 1;
  hidden_kernel<<<n, 256, 0, stream>>>(seed, seq, layer, pos0, n, D, scale, drift, seg_amp, inv_sd, d_mean, d_seg,
                                      static_cast<uint16_t*>(d_out), row_stride);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// K and V rows of positions pos0..pos0+n-1 written to slots slot0..slot0+n-1.
int synth_kv(uint64_t seed, int seq, int pos0, int n, int slot0, int L, int H, int d, int spike_per_10k,
             const float* d_kv_scale, const float* d_kv_off, void* k, void* v, int layout, int64_t stride_layer,
             int64_t stride_seq, int64_t stride_block, int64_t stride_token, const int32_t* block_table,
             int max_blocks, int block_size, cudaStream_t stream) {
  if (n <= 0) return 0;
  if (d % 8 || H * d / 8 > 1024 || !k || !v) return 1;
  View vw;
  vw.base[0] = static_cast<char*>(k);
  vw.base[1] = static_cast<char*>(v);
  vw.layout = layout;
  vw.stride_layer = stride_layer;
  vw.stride_seq = stride_seq;
  vw.stride_block = stride_block;
  vw.stride_token = stride_token;
  vw.block_table = block_table;
  vw.max_blocks = max_blocks;
  vw.block_size = block_size;
  dim3 grid(n, L, 2);
  const int threads = (H * d / 8 + 31) / 32 * 32;
  kv_kernel<<<grid, threads, 0, stream>>>(seed, seq, pos0, n, slot0, L, H, d, spike_per_10k, d_kv_scale, d_kv_off, vw);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// Batched hidden rows of one layer: row i of d_out is (d_seqs[i], d_pos[i]).
int synth_hidden_batch(uint64_t seed, int layer, int n, const int32_t* d_seqs, const int32_t* d_pos, int D,
                       float scale, float drift, float seg_amp, float inv_sd, const float* d_mean,
                       const int32_t* d_seg, int64_t seg_stride, void* d_out, int64_t row_stride,
                       cudaStream_t stream) {
  if (n <= 0) return 0;
  if (D % 8 || !d_mean || !d_out || !d_seqs || !d_pos || (seg_amp != 0.0f && !d_seg)) return 1;
  hidden_batch_kernel<<<n, 256, 0, stream>>>(seed, layer, n, d_seqs, d_pos, D, scale, drift, seg_amp, inv_sd, d_mean,
                                            d_seg, seg_stride, static_cast<uint16_t*>(d_out), row_stride);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

// Batched K/V rows: (d_seqs[i], d_pos[i]) written to slot d_slots[i] of sequence d_seqs[i].
int synth_kv_batch(uint64_t seed, int n, const int32_t* d_seqs, const int32_t* d_pos, const int32_t* d_slots, int L,
                   int H, int d, int spike_per_10k, const float* d_kv_scale, const float* d_kv_off, void* k, void* v,
                   int layout, int64_t stride_layer, int64_t stride_seq, int64_t stride_block, int64_t stride_token,
                   const int32_t* block_table, int max_blocks, int block_size, cudaStream_t stream) {
  if (n <= 0) return 0;
  if (d % 8 || H * d / 8 > 1024 || !k || !v || !d_seqs || !d_pos || !d_slots) return 1;
  View vw;
  vw.base[0] = static_cast<char*>(k);
  vw.base[1] = static_cast<char*>(v);
  vw.layout = layout;
  vw.stride_layer = stride_layer;
  vw.stride_seq = stride_seq;
  vw.stride_block = stride_block;
  vw.stride_token = stride_token;
  vw.block_table = block_table;
  vw.max_blocks = max_blocks;
  vw.block_size = block_size;
  dim3 grid(n, L, 2);
  const int threads = (H * d / 8 + 31) / 32 * 32;
  kv_batch_kernel<<<grid, threads, 0, stream>>>(seed, n, d_seqs, d_pos, d_slots, L, H, d, spike_per_10k, d_kv_scale,
                                                d_kv_off, vw);
  return cudaGetLastError() == cudaSuccess ? 0 : 2;
}

}  // extern "C"
