// C ABI of libepikv: argument validation, workspace carving and launch
// sequencing.  No entry point allocates device memory; epikv_init allocates
// the host-side context only.
#include <stdlib.h>
#include <string.h>

#include "common.cuh"
#include "kernels.h"

using namespace epikv;

struct epikv_ctx {
  epikv_config cfg;
  Dims dm;
  DevState st;
  void* ws;
  size_t ws_bytes;
  int device;
  int num_sms;
  int compact_ctas;
  cudaStream_t last_stream;
  bool timing;
  cudaEvent_t ev[4];
  bool kclock_on;
  KernelClock kclock;   // per-kernel events (epikv_set_kernel_events)
};

namespace {

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

int next_pow2(int x) {
  int p = 1;
  while (p < x) p <<= 1;
  return p;
}

bool is_pow2(int x) { return x > 0 && (x & (x - 1)) == 0; }

bool valid_config(const epikv_config* c) {
  if (!c) return false;
  if (c->max_seqs < 1 || c->max_seqs > 4096) return false;
  if (c->max_cache_tokens < 1 || c->max_cache_tokens > (1 << 24)) return false;
  if (c->max_new_tokens < 1 || c->max_new_tokens > (1 << 20)) return false;
  if (c->score_kinds < 1 || c->score_kinds > 63) return false;
  if (c->recency_cap < 0) return false;
  if (c->select_chunk < 0 || c->select_chunk > 65536) return false;
  if (c->layer_budgets != 0 && c->layer_budgets != 1) return false;
  if (c->layer_budgets && (c->num_layers > 64 || c->select_chunk > 1)) return false;
  if (c->num_layers < 1 || c->num_kv_heads < 1 || c->num_kv_heads > 32) return false;
  if (!is_pow2(c->head_dim) || c->head_dim < 8 || c->head_dim > 256) return false;
  if (c->num_kv_heads * c->head_dim / 8 > 256) return false;
  if (c->score_kinds & kBandKinds) {
    if (c->hidden < 8 || c->hidden % 8 != 0 || c->hidden > 8192) return false;
    if (c->n_band_a < 1 || c->n_band_b < 1 || c->n_band_a + c->n_band_b > kMaxBand) return false;
    if (c->z_window < 1 || c->z_window > 1024 || !(c->z_eps >= 0.f)) return false;
  }
  if (c->score_kinds & kKvKinds) {
    if (c->lag < 1 || c->lag_window < 1 || c->lag_window > 1024 || !(c->lag_eps >= 0.f)) return false;
    if ((int64_t)c->max_new_tokens * 2 * c->num_layers > (int64_t)1 << 30) return false;
  }
  return true;
}

Dims make_dims(const epikv_config* c) {
  Dims d;
  memset(&d, 0, sizeof(d));
  d.S = c->max_seqs;
  d.T = c->max_cache_tokens;
  d.max_new = c->max_new_tokens;
  d.L = c->num_layers;
  d.H = c->num_kv_heads;
  d.d = c->head_dim;
  d.kinds = c->score_kinds;
  d.recency_cap = c->recency_cap;
  d.select_chunk = c->select_chunk > 1 ? c->select_chunk : 1;
  d.layer_budgets = c->layer_budgets;
  const bool bz = c->score_kinds & kBandKinds, lg = c->score_kinds & kKvKinds;
  d.D = bz ? c->hidden : 0;
  d.nA = bz ? c->n_band_a : 0;
  d.nB = bz ? c->n_band_b : 0;
  d.z_window = bz ? c->z_window : 1;
  d.z_eps = c->z_eps;
  d.lag = lg ? c->lag : 1;
  d.lag_window = lg ? c->lag_window : 1;
  d.lag_eps = c->lag_eps;
  // rings hold every position a window of this call can reach (see finalize)
  d.stash_rows = d.T < kStashRows ? d.T : kStashRows;
  d.G = next_pow2(c->max_new_tokens + (d.z_window > d.lag_window ? d.z_window : d.lag_window));
  return d;
}

// Lay the state out in `base` (nullptr: only size it).  256-byte aligned.
size_t carve(const Dims& d, DevState* st, char* base) {
  size_t off = 0;
  auto take = [&](size_t bytes) -> void* {
    off = align_up(off, 256);
    void* p = base ? base + off : nullptr;
    off += bytes;
    return p;
  };
  const size_t S = d.S, T = d.T;
  memset(st, 0, sizeof(*st));
  st->n_cache = (int32_t*)take(S * 4);
  st->n_seen = (int32_t*)take(S * 4);
  st->prefill = (int32_t*)take(S * 4);
  st->policy = (int32_t*)take(S * 4);
  st->hp_parity = (int32_t*)take(S * 4);
  st->first_changed = (int32_t*)take(S * 4);
  st->ticket = (uint32_t*)take(S * 4);
  st->err = (int32_t*)take(4);
  st->stats = (unsigned long long*)take(4 * 8);
  st->pos = (int32_t*)take(S * T * 4);
  const size_t LB = d.layer_budgets ? (size_t)d.L : 1;  // kept lists and lengths per layer
  st->kept = (int32_t*)take(S * LB * T * 4);
  st->n_kept = (int32_t*)take(S * LB * 4);
  for (int k = 0; k < kNumKinds; ++k)
    if (d.kinds & (1 << k)) st->score[k] = (float*)take(S * T * 4);
  if (d.kinds & kBandKinds) {
    const size_t nb = d.nA + d.nB;
    st->h_prev = (__nv_bfloat16*)take(S * 2 * nb * d.D * 2);
    st->g_ring = (float*)take(S * nb * d.G * 4);
    st->ztok = (float*)take(S * 2 * nb * 4);
  }
  if (d.kinds & kNormKinds) {
    st->lag_rng = (__nv_bfloat16*)take(S * d.L * 2 * 4 * (size_t)d.H * d.d * 2);
    st->lag_part = (float*)take(S * (size_t)d.max_new * 2 * d.L * 4);
  }
  if (d.kinds & kRawKinds) st->raw_part = (float*)take(S * (size_t)d.max_new * 2 * d.L * 4);
  for (int q = 0; q < 4; ++q)
    if (d.kinds & kv_kind(q)) st->u_ring[q] = (float*)take(S * (size_t)d.G * 4);
  if (d.select_chunk > 1) st->ckey = (uint32_t*)take(S * T * 4);
  if (d.layer_budgets) {
    st->n_layer = (int32_t*)take(S * d.L * 4);
    st->lfirst = (int32_t*)take(S * d.L * 4);
    st->lmask = (unsigned long long*)take(S * T * 8);
    st->lmask_new = (unsigned long long*)take(S * T * 8);
    st->lkeep = (uint32_t*)take(S * d.L * ((T + 31) / 32) * 4);
    st->mkept = (int32_t*)take(S * T * 4);
  }
  st->work = (uint32_t*)take(2 * 4);
  st->stash = (char*)take((size_t)kMaxStashCtas * d.stash_rows * d.H * d.d * 2);
  st->stash_row0 = (int32_t*)take((size_t)kMaxStashCtas * 4);
  return align_up(off, 256);
}

bool aligned16(const void* p) { return ((uintptr_t)p & 15u) == 0; }

bool valid_kv(const epikv_ctx* ctx, const epikv_kv_view* kv, KvDev* out) {
  if (!kv || !kv->k || !kv->v || !aligned16(kv->k) || !aligned16(kv->v)) return false;
  const int64_t hd = (int64_t)ctx->dm.H * ctx->dm.d;
  if (kv->stride_token < hd || kv->stride_token % 8 || kv->stride_layer < 0 || kv->stride_layer % 8) return false;
  memset(out, 0, sizeof(*out));
  out->base[0] = (char*)kv->k;
  out->base[1] = (char*)kv->v;
  out->layout = kv->layout;
  out->stride_layer = kv->stride_layer;
  out->stride_token = kv->stride_token;
  if (kv->layout == EPIKV_LAYOUT_CONTIGUOUS) {
    if (kv->stride_seq < 0 || kv->stride_seq % 8) return false;
    out->stride_seq = kv->stride_seq;
    return true;
  }
  if (kv->layout != EPIKV_LAYOUT_PAGED) return false;
  if (!kv->block_table || kv->block_size < 1 || kv->max_blocks_per_seq < 1 || kv->num_blocks < 1) return false;
  if (kv->stride_block < 0 || kv->stride_block % 8 || kv->stride_table_layer < 0) return false;
  out->stride_block = kv->stride_block;
  out->table_stride_layer = kv->stride_table_layer;
  out->block_table = kv->block_table;
  out->max_blocks = kv->max_blocks_per_seq;
  out->block_size = kv->block_size;
  out->num_blocks = kv->num_blocks;
  return true;
}

bool valid_hidden(const epikv_ctx* ctx, const epikv_hidden_view* hv) {
  if (!(ctx->dm.kinds & kBandKinds)) return true;
  if (!hv || hv->row_stride < ctx->dm.D || hv->row_stride % 8) return false;
  for (int i = 0; i < ctx->dm.nA + ctx->dm.nB; ++i)
    if (!hv->band_rows[i] || !aligned16(hv->band_rows[i])) return false;
  return true;
}

epikv_status cuda_status(cudaError_t e) { return e == cudaSuccess ? EPIKV_OK : EPIKV_ECUDA; }

// Points the launch helpers at the context's kernel events (if set) for the
// duration of one entry point.
struct ClockScope {
  explicit ClockScope(epikv_ctx* ctx) { t_kernel_clock = ctx && ctx->kclock_on ? &ctx->kclock : nullptr; }
  ~ClockScope() { t_kernel_clock = nullptr; }
};

}  // namespace

extern "C" {

size_t epikv_workspace_bytes(const epikv_config* cfg) {
  if (!valid_config(cfg)) return 0;
  DevState st;
  return carve(make_dims(cfg), &st, nullptr);
}

epikv_status epikv_init(epikv_ctx** out, const epikv_config* cfg, void* d_workspace, size_t workspace_bytes,
                        cudaStream_t stream) {
  if (!out || !valid_config(cfg) || !d_workspace || ((uintptr_t)d_workspace & 255u)) return EPIKV_EINVAL;
  *out = nullptr;
  const size_t need = epikv_workspace_bytes(cfg);
  if (workspace_bytes < need) return EPIKV_EINVAL;
  epikv_ctx* ctx = (epikv_ctx*)calloc(1, sizeof(epikv_ctx));
  if (!ctx) return EPIKV_EINVAL;
  ctx->cfg = *cfg;
  ctx->dm = make_dims(cfg);
  carve(ctx->dm, &ctx->st, (char*)d_workspace);
  ctx->ws = d_workspace;
  ctx->ws_bytes = workspace_bytes;
  ctx->last_stream = stream;
  cudaError_t e = cudaGetDevice(&ctx->device);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->device);
  int per_sm = 1;
  if (e == cudaSuccess) e = compact_prepare(ctx->device, &per_sm);
  if (e == cudaSuccess) e = finalize_prepare();
  if (e == cudaSuccess) e = select_prepare();
  ctx->compact_ctas = ctx->num_sms * per_sm;
  if (e == cudaSuccess) e = cudaMemsetAsync(d_workspace, 0, need, stream);
  if (e == cudaSuccess) e = launch_init_state(ctx->st, ctx->dm, stream);
  if (e != cudaSuccess) {
    free(ctx);
    return EPIKV_ECUDA;
  }
  *out = ctx;
  return EPIKV_OK;
}

epikv_status epikv_seq_reset(epikv_ctx* ctx, int32_t seq, int32_t prefill_len, int32_t policy,
                             cudaStream_t stream) {
  if (!ctx || seq < 0 || seq >= ctx->dm.S || prefill_len < 0) return EPIKV_EINVAL;
  if (policy < 1 || (policy & (policy - 1)) || !(policy & ctx->dm.kinds)) return EPIKV_EINVAL;
  ctx->last_stream = stream;
  return cuda_status(launch_reset_seq(ctx->st, ctx->dm, seq, prefill_len, policy, stream));
}

static epikv_status score_update_impl(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids,
                                      const int32_t* d_cu_new, int32_t max_new,
                                      const epikv_hidden_view* hidden, const epikv_kv_view* kv,
                                      cudaStream_t stream, int* launches) {
  if (!ctx || n_seq < 0 || n_seq > ctx->dm.S || max_new < 0 || max_new > ctx->dm.max_new) return EPIKV_EINVAL;
  if (n_seq == 0) return EPIKV_OK;  // nothing to score
  if (!d_seq_ids || !d_cu_new) return EPIKV_EINVAL;
  if (!valid_hidden(ctx, hidden)) return EPIKV_EINVAL;
  KvDev kd;
  memset(&kd, 0, sizeof(kd));
  if ((ctx->dm.kinds & kKvKinds) && !valid_kv(ctx, kv, &kd)) return EPIKV_EINVAL;
  ctx->last_stream = stream;
  return cuda_status(launch_score_update(ctx->st, ctx->dm, n_seq, d_seq_ids, d_cu_new, max_new, hidden, &kd,
                                         ctx->num_sms, stream, launches));
}

epikv_status epikv_score_update(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids, const int32_t* d_cu_new,
                                int32_t max_new, const epikv_hidden_view* hidden, const epikv_kv_view* kv,
                                cudaStream_t stream) {
  int launches = 0;
  ClockScope clock(ctx);
  return score_update_impl(ctx, n_seq, d_seq_ids, d_cu_new, max_new, hidden, kv, stream, &launches);
}

epikv_status epikv_select(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids, const int32_t* d_budget,
                          const int32_t* d_trigger, int32_t* d_kept, int32_t kept_stride, int32_t* d_n_kept,
                          cudaStream_t stream) {
  if (!ctx || n_seq < 0 || n_seq > ctx->dm.S || kept_stride < 1) return EPIKV_EINVAL;
  if (n_seq > 0 && (!d_seq_ids || !d_budget || !d_kept)) return EPIKV_EINVAL;
  ctx->last_stream = stream;
  int launches = 0;
  ClockScope clock(ctx);
  return cuda_status(launch_select(ctx->st, ctx->dm, n_seq, d_seq_ids, d_budget, d_trigger, d_kept, kept_stride,
                                   d_n_kept, stream, &launches));
}

epikv_status epikv_compact(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids, const int32_t* d_kept,
                           int32_t kept_stride, const epikv_kv_view* kv, cudaStream_t stream) {
  if (!ctx || n_seq < 0 || n_seq > ctx->dm.S || kept_stride < 1) return EPIKV_EINVAL;
  if (n_seq > 0 && (!d_seq_ids || !d_kept)) return EPIKV_EINVAL;
  KvDev kd;
  if (!valid_kv(ctx, kv, &kd)) return EPIKV_EINVAL;
  ctx->last_stream = stream;
  int launches = 0;
  ClockScope clock(ctx);
  return cuda_status(
      launch_compact(ctx->st, ctx->dm, n_seq, d_seq_ids, d_kept, kept_stride, kd, ctx->compact_ctas, stream, &launches));
}

epikv_status epikv_step(epikv_ctx* ctx, int32_t n_seq, const int32_t* d_seq_ids, const int32_t* d_cu_new,
                        int32_t max_new, const int32_t* d_budget, const int32_t* d_trigger,
                        const epikv_hidden_view* hidden, const epikv_kv_view* kv, int32_t* d_n_cache_out,
                        cudaStream_t stream) {
  if (!ctx || n_seq < 0 || n_seq > ctx->dm.S) return EPIKV_EINVAL;
  if (n_seq == 0) return EPIKV_OK;  // nothing to do
  if (!d_budget) return EPIKV_EINVAL;
  KvDev kd;
  if (!valid_kv(ctx, kv, &kd)) return EPIKV_EINVAL;
  int launches = 0;
  ClockScope clock(ctx);
  cudaError_t e = cudaSuccess;
  if (ctx->timing) e = cudaEventRecord(ctx->ev[0], stream);
  if (e != cudaSuccess) return EPIKV_ECUDA;
  epikv_status s = score_update_impl(ctx, n_seq, d_seq_ids, d_cu_new, max_new, hidden, kv, stream, &launches);
  if (s != EPIKV_OK) return s;
  if (ctx->timing) e = cudaEventRecord(ctx->ev[1], stream);
  if (e == cudaSuccess)
    e = launch_select(ctx->st, ctx->dm, n_seq, d_seq_ids, d_budget, d_trigger, ctx->st.kept, ctx->dm.T,
                      d_n_cache_out ? d_n_cache_out : ctx->st.n_kept, stream, &launches);
  if (e == cudaSuccess && ctx->timing) e = cudaEventRecord(ctx->ev[2], stream);
  if (e == cudaSuccess)
    e = launch_compact(ctx->st, ctx->dm, n_seq, d_seq_ids, ctx->st.kept, ctx->dm.T, kd, ctx->compact_ctas, stream,
                       &launches);
  if (e == cudaSuccess && ctx->timing) e = cudaEventRecord(ctx->ev[3], stream);
  return cuda_status(e);
}

epikv_status epikv_set_phase_events(epikv_ctx* ctx, const cudaEvent_t* events) {
  if (!ctx) return EPIKV_EINVAL;
  if (!events) {
    ctx->timing = false;
    return EPIKV_OK;
  }
  for (int i = 0; i < 4; ++i) {
    if (!events[i]) return EPIKV_EINVAL;
    ctx->ev[i] = events[i];
  }
  ctx->timing = true;
  return EPIKV_OK;
}

epikv_status epikv_set_kernel_events(epikv_ctx* ctx, const cudaEvent_t* events, int32_t n_kernels,
                                     const char** h_names, int32_t* h_used) {
  if (!ctx) return EPIKV_EINVAL;
  if (!events) {
    if (h_used) *h_used = ctx->kclock_on ? ctx->kclock.used : 0;
    ctx->kclock_on = false;
    return EPIKV_OK;
  }
  if (n_kernels < 1 || !h_names) return EPIKV_EINVAL;
  for (int i = 0; i < 2 * n_kernels; ++i)
    if (!events[i]) return EPIKV_EINVAL;
  for (int i = 0; i < n_kernels; ++i) h_names[i] = nullptr;
  ctx->kclock.ev = const_cast<cudaEvent_t*>(events);
  ctx->kclock.names = h_names;
  ctx->kclock.cap = n_kernels;
  ctx->kclock.used = 0;
  ctx->kclock_on = true;
  if (h_used) *h_used = 0;
  return EPIKV_OK;
}

epikv_status epikv_read_slots(epikv_ctx* ctx, int32_t seq, int32_t kind, float* h_score, int32_t* h_pos,
                              int32_t cap, int32_t* h_n) {
  if (!ctx || seq < 0 || seq >= ctx->dm.S || cap < 0 || !h_n) return EPIKV_EINVAL;
  if (h_score && (kind < 1 || (kind & (kind - 1)) || !(kind & ctx->dm.kinds))) return EPIKV_EINVAL;
  cudaError_t e = cudaStreamSynchronize(ctx->last_stream);
  int32_t n = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&n, ctx->st.n_cache + seq, 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return EPIKV_ECUDA;
  *h_n = n;
  const int m = n < cap ? n : cap;
  if (m > 0 && h_pos)
    e = cudaMemcpy(h_pos, ctx->st.pos + (size_t)seq * ctx->dm.T, (size_t)m * 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && m > 0 && h_score)
    e = cudaMemcpy(h_score, ctx->st.score[kind_index(kind)] + (size_t)seq * ctx->dm.T, (size_t)m * 4,
                   cudaMemcpyDeviceToHost);
  return cuda_status(e);
}

epikv_status epikv_read_layer_slots(epikv_ctx* ctx, int32_t seq, int32_t layer, int32_t* h_pos, int32_t cap,
                                    int32_t* h_n) {
  if (!ctx || !ctx->dm.layer_budgets || seq < 0 || seq >= ctx->dm.S || layer < 0 || layer >= ctx->dm.L || cap < 0 ||
      !h_n)
    return EPIKV_EINVAL;
  cudaError_t e = cudaStreamSynchronize(ctx->last_stream);
  int32_t n = 0;
  if (e == cudaSuccess) e = cudaMemcpy(&n, ctx->st.n_cache + seq, 4, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return EPIKV_ECUDA;
  int32_t* pos = (int32_t*)malloc((size_t)(n > 0 ? n : 1) * 4);
  unsigned long long* mask = (unsigned long long*)malloc((size_t)(n > 0 ? n : 1) * 8);
  if (!pos || !mask) {
    free(pos);
    free(mask);
    return EPIKV_EINVAL;
  }
  const size_t base = (size_t)seq * ctx->dm.T;
  if (n > 0) e = cudaMemcpy(pos, ctx->st.pos + base, (size_t)n * 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && n > 0) e = cudaMemcpy(mask, ctx->st.lmask + base, (size_t)n * 8, cudaMemcpyDeviceToHost);
  int32_t nl = 0;
  if (e == cudaSuccess)
    for (int i = 0; i < n; ++i)
      if ((mask[i] >> layer) & 1ull) {
        if (h_pos && nl < cap) h_pos[nl] = pos[i];
        ++nl;
      }
  free(pos);
  free(mask);
  *h_n = nl;
  return cuda_status(e);
}

epikv_status epikv_get_stats(epikv_ctx* ctx, epikv_stats* out) {
  if (!ctx || !out) return EPIKV_EINVAL;
  cudaError_t e = cudaStreamSynchronize(ctx->last_stream);
  if (e == cudaSuccess) e = cudaMemcpy(out, ctx->st.stats, sizeof(epikv_stats), cudaMemcpyDeviceToHost);
  return cuda_status(e);
}

epikv_status epikv_get_error(epikv_ctx* ctx, int32_t* code) {
  if (!ctx) return EPIKV_EINVAL;
  int32_t v = 0;
  cudaError_t e = cudaStreamSynchronize(ctx->last_stream);
  if (e == cudaSuccess) e = cudaMemcpy(&v, ctx->st.err, 4, cudaMemcpyDeviceToHost);
  if (e == cudaSuccess && v != 0) e = cudaMemset(ctx->st.err, 0, 4);
  if (e != cudaSuccess) return EPIKV_ECUDA;
  if (code) *code = v;
  return v ? EPIKV_EDEVICE : EPIKV_OK;
}

void epikv_destroy(epikv_ctx* ctx) { free(ctx); }

const char* epikv_status_string(epikv_status s) {
  switch (s) {
    case EPIKV_OK: return "ok";
    case EPIKV_EINVAL: return "invalid argument";
    case EPIKV_ECUDA: return "CUDA error";
    case EPIKV_EDEVICE: return "device-side error";
  }
  return "unknown status";
}

}  // extern "C"
