// Device-side helpers shared by the EpiKV kernels: the context's device
// state, K/V row addressing for both layouts, the sticky error word, and
// inline-PTX wrappers for 1-D TMA bulk copies and mbarriers (sm_90+ ISA,
// compiled here for sm_103a only).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "epikv.h"

namespace epikv {

constexpr int kMaxBand = 32;
constexpr int kNumKinds = 6;  // score kind index k <-> mask bit (1 << k)
constexpr int kBandKinds = EPIKV_SCORE_BANDZ | EPIKV_SCORE_HSVAR;
constexpr int kNormKinds = EPIKV_SCORE_LAGKV | EPIKV_SCORE_LAGKEY;   // need the chunk ranges
constexpr int kRawKinds = EPIKV_SCORE_KVKEY | EPIKV_SCORE_KVVAL;
constexpr int kKvKinds = kNormKinds | kRawKinds;
// the K/V kinds in the order of their rolling-mean rings
__host__ __device__ __forceinline__ int kv_kind(int q) {
  return q == 0 ? EPIKV_SCORE_LAGKV : q == 1 ? EPIKV_SCORE_KVKEY : q == 2 ? EPIKV_SCORE_KVVAL : EPIKV_SCORE_LAGKEY;
}

__host__ __device__ __forceinline__ int kind_index(int bit) {
  int k = 0;
  while (bit > 1) {
    bit >>= 1;
    ++k;
  }
  return k;
}

// Device pointers carved out of the caller's workspace (one context).
struct DevState {
  int32_t* n_cache;        // [S] slots in use
  int32_t* n_seen;         // [S] next position
  int32_t* prefill;        // [S]
  int32_t* policy;         // [S] score kind driving selection (1 or 2)
  int32_t* hp_parity;      // [S] which h_prev buffer holds the last row
  int32_t* first_changed;  // [S] first slot moved by the last selection
  uint32_t* ticket;        // [S] last-CTA tickets of the finalize kernel
  int32_t* err;            // [1] sticky device error word
  unsigned long long* stats;  // [4] epikv_stats
  float* score[kNumKinds]; // [S][T] frozen scores per kind (null when the kind is off)
  int32_t* pos;            // [S][T] position of each slot
  __nv_bfloat16* h_prev;   // [S][2][n_band][D] last hidden row per band layer
  float* g_ring;           // [S][n_band][G] g by position (mod G)
  float* ztok;             // [S][2][n_band] a decode step's per-band z and window mean of g (band kinds)
  __nv_bfloat16* lag_rng;  // [S][L][2][4][H][d] prev min, prev max, cur min, cur max
  float* lag_part;         // [S][max_new][2L] per-(layer, K|V) head-summed normalised variances
  float* raw_part;         // [S][max_new][2L] per-(layer, K|V) head-summed raw variances
  float* u_ring[4];        // [S][G] per K/V kind (kv_kind order): u by position (mod G)
  int32_t* kept;           // [S][T] kept lists of epikv_step
  int32_t* n_kept;         // [S]
  uint32_t* ckey;          // [S][T] chunk-level selection: each candidate slot's chunk key (C > 1 only)
  // per-layer budgets only (null otherwise)
  int32_t* n_layer;        // [S][L] slots held by each layer
  int32_t* lfirst;         // [S][L] first slot of each layer moved by the last selection
  unsigned long long* lmask;      // [S][T] bit l: layer l holds the token of this slot
  unsigned long long* lmask_new;  // [S][T] the select kernel's new masks (scratch)
  uint32_t* lkeep;         // [S][L][ceil(T/32)] bit: layer l keeps the union slot (scratch)
  int32_t* mkept;          // [S][T] the select kernel's kept slots of the largest layer (scratch)
  uint32_t* work;          // [2] the compaction's next unit (per-layer budgets) and finished CTAs (0 between launches)
  char* stash;             // [kMaxStashCtas][stash_rows][H*d] bf16: compaction boundary rows (token budgets)
  int32_t* stash_row0;     // [kMaxStashCtas] the row whose source is each stash's first row
};

// The balanced compaction split: at most this many CTAs, each with a stash
// of at most kStashRows rows (the slots its left neighbour still reads).
constexpr int kMaxStashCtas = 512;
constexpr int kStashRows = 128;

struct Dims {
  int S, T, max_new, L, H, d, D, nA, nB, G;
  int stash_rows;  // min(kStashRows, T): rows of one CTA's compaction stash
  int z_window, lag, lag_window, recency_cap, kinds, select_chunk, layer_budgets;
  float z_eps, lag_eps;
};

struct KvDev {
  char* base[2];           // K, V
  int layout;
  int64_t stride_layer, stride_seq, stride_block, stride_token;  // elements
  const int32_t* block_table;
  int max_blocks, block_size, num_blocks;
  int64_t table_stride_layer;  // elements between layers' block tables (0: shared)
};

// Programmatic dependent launch.  The kernels of a step are launched with
// programmatic stream serialisation (pdl_launch): each may be scheduled while
// the kernel before it on the stream finishes, and waits in pdl_wait -- its
// first statement -- until that kernel has completed and its writes are
// visible; pdl_trigger lets the next kernel be scheduled once every CTA of
// this one has started.  Launched without the attribute, both are no-ops.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

#ifndef EPIKV_PDL
#define EPIKV_PDL 1  // 0: plain stream order
#endif

template <typename... Params, typename... Args>
inline cudaError_t launch_kernel_now(bool programmatic, void (*kernel)(Params...), dim3 grid, dim3 block,
                                     size_t smem, cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = programmatic && EPIKV_PDL ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// Per-kernel timing (epikv_set_kernel_events): while an entry point of a
// context with kernel events runs, t_kernel_clock points at its record, and
// every kernel it launches is bracketed by two of the caller's events on the
// launch stream, its name (cudaFuncGetName) stored beside them.
struct KernelClock {
  cudaEvent_t* ev;      // [2 * cap]: before and after each kernel
  const char** names;   // [cap]
  int cap, used;
};
inline thread_local KernelClock* t_kernel_clock = nullptr;

template <typename... Params, typename... Args>
inline cudaError_t launch_kernel(bool programmatic, void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                                 cudaStream_t stream, Args... args) {
  KernelClock* kc = t_kernel_clock;
  if (kc && kc->used < kc->cap) {
    const cudaError_t e = cudaEventRecord(kc->ev[2 * kc->used], stream);
    if (e != cudaSuccess) return e;
  } else {
    kc = nullptr;
  }
  const cudaError_t e = launch_kernel_now(programmatic, kernel, grid, block, smem, stream, args...);
  if (e != cudaSuccess || !kc) return e;
  const char* name = nullptr;
  if (cudaFuncGetName(&name, reinterpret_cast<const void*>(kernel)) != cudaSuccess) name = nullptr;
  kc->names[kc->used] = name;
  return cudaEventRecord(kc->ev[2 * kc->used++ + 1], stream);
}


template <typename... Params, typename... Args>
inline cudaError_t pdl_launch(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                              Args... args) {
  return launch_kernel(true, kernel, grid, block, smem, stream, args...);
}

// Plain stream order: the long copy kernel, whose CTAs spread more evenly
// when none of them is placed before the kernel ahead of it has finished.
template <typename... Params, typename... Args>
inline cudaError_t plain_launch(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                                Args... args) {
  return launch_kernel(false, kernel, grid, block, smem, stream, args...);
}

__device__ __forceinline__ void set_error(int32_t* err, int code) {
  atomicCAS(err, 0, code);
}

// Element offset of (layer, seq, slot) or -1 if outside the view.
__device__ __forceinline__ int64_t kv_row_offset(const KvDev& v, int layer, int seq, int slot, int T) {
  if (slot < 0) return -1;
  if (v.layout == EPIKV_LAYOUT_CONTIGUOUS) {
    if (slot >= T) return -1;
    return (int64_t)layer * v.stride_layer + (int64_t)seq * v.stride_seq + (int64_t)slot * v.stride_token;
  }
  int bi = slot / v.block_size;
  if (bi >= v.max_blocks) return -1;
  int blk = __ldg(v.block_table + (int64_t)layer * v.table_stride_layer + (int64_t)seq * v.max_blocks + bi);
  if (blk < 0 || blk >= v.num_blocks) return -1;
  return (int64_t)layer * v.stride_layer + (int64_t)blk * v.stride_block +
         (int64_t)(slot - bi * v.block_size) * v.stride_token;
}

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ void unpack8(const uint4& q, float* f) {
  f[0] = bf16_lo(q.x); f[1] = bf16_hi(q.x);
  f[2] = bf16_lo(q.y); f[3] = bf16_hi(q.y);
  f[4] = bf16_lo(q.z); f[5] = bf16_hi(q.z);
  f[6] = bf16_lo(q.w); f[7] = bf16_hi(q.w);
}

// Streaming 16-byte load that does not allocate in L1.
__device__ __forceinline__ uint4 ld_stream16(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "l"(p));
  return r;
}

// The same load when `take`, else zeros: a predicated instruction, no branch.
__device__ __forceinline__ uint4 ld_stream16_if(const void* p, bool take) {
  uint4 r = make_uint4(0, 0, 0, 0);
  asm volatile(
      "{\n\t.reg .pred q;\n\tsetp.ne.b32 q, %5, 0;\n\t"
      "@q ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];\n\t}"
      : "+r"(r.x), "+r"(r.y), "+r"(r.z), "+r"(r.w) : "l"(p), "r"((int)take));
  return r;
}

// ---------------------------------------------------------------- mbarrier
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_u32(bar)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.release.cta.shared::cta.b64 _, [%0], %1;"
               :: "r"(smem_u32(bar)), "r"(bytes) : "memory");
}

#ifndef EPIKV_MBAR_SPIN
#define EPIKV_MBAR_SPIN 2
#endif

// One probe; true when the phase with `parity` has completed.  The default
// (2) may suspend the thread for a short, hardware-chosen time; 1 polls
// without suspending; 0 asks for a suspension of up to 1 us.
__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
#if EPIKV_MBAR_SPIN == 1
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.test_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
#elif EPIKV_MBAR_SPIN == 2
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
#else
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cta.shared::cta.b64 p, [%1], %2, 1000;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok) : "r"(smem_u32(bar)), "r"(parity) : "memory");
#endif
  return ok != 0;
}

__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait at most `limit_ns` of wall time; false if it gave up.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  while (!mbar_try_wait(bar, parity))
    if (global_ns() - t0 > limit_ns) return false;
  return true;
}

__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ------------------------------------------------------------ TMA bulk copies
// global -> shared, completion counted in bytes on `bar`.
__device__ __forceinline__ void tma_load_1d(void* smem_dst, const void* gmem_src, uint32_t bytes, uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
      :: "r"(smem_u32(smem_dst)), "l"(gmem_src), "r"(bytes), "r"(smem_u32(bar)) : "memory");
}

// shared -> global, tracked by this thread's bulk async-groups.
__device__ __forceinline__ void tma_store_1d(void* gmem_dst, const void* smem_src, uint32_t bytes) {
  asm volatile("cp.async.bulk.global.shared::cta.bulk_group [%0], [%1], %2;"
               :: "l"(gmem_dst), "r"(smem_u32(smem_src)), "r"(bytes) : "memory");
}

__device__ __forceinline__ void tma_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }

// Wait until at most N of this thread's bulk groups still read shared memory.
template <int N>
__device__ __forceinline__ void tma_wait_read() {
  asm volatile("cp.async.bulk.wait_group.read %0;" :: "n"(N) : "memory");
}

__device__ __forceinline__ void tma_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// ------------------------------------------------------------ warp helpers
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over aligned groups of `width` lanes (width a power of two <= 32).
__device__ __forceinline__ float group_sum(float v, int width) {
  for (int o = width >> 1; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

}  // namespace epikv
