// Host-side launchers of the EpiKV kernels (internal to libepikv).
#pragma once

#include "common.cuh"

namespace epikv {

// Band-z g kernel (if enabled), Lag-KV partial kernel (if enabled) and the
// finalize kernel; *launches is incremented per kernel launched.
cudaError_t launch_score_update(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                                const int32_t* cu_new, int max_new, const epikv_hidden_view* hv,
                                const KvDev* kv, int num_sms, cudaStream_t stream, int* launches);

cudaError_t launch_select(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                          const int32_t* budget, const int32_t* trigger, int32_t* kept, int kept_stride,
                          int32_t* n_kept, cudaStream_t stream, int* launches);

// Grid of `ctas` persistent CTAs (0: the library's choice for this device).
cudaError_t launch_compact(const DevState& st, const Dims& dm, int n_seq, const int32_t* seq_ids,
                           const int32_t* kept, int kept_stride, const KvDev& kv, int ctas,
                           cudaStream_t stream, int* launches);

cudaError_t compact_prepare(int device, int* ctas_per_sm);
cudaError_t finalize_prepare();
cudaError_t select_prepare();

cudaError_t launch_reset_seq(const DevState& st, const Dims& dm, int seq, int prefill, int policy,
                             cudaStream_t stream);
cudaError_t launch_init_state(const DevState& st, const Dims& dm, cudaStream_t stream);

}  // namespace epikv
