// Small state kernels: context initialisation and per-sequence reset.
#include "common.cuh"
#include "kernels.h"

namespace epikv {

__global__ void init_state_kernel(DevState st, Dims dm) {
  const int default_policy = dm.kinds & -dm.kinds;  // the lowest enabled kind
  for (int s = blockIdx.x * blockDim.x + threadIdx.x; s < dm.S; s += gridDim.x * blockDim.x)
    st.policy[s] = default_policy;
}

__global__ void reset_seq_kernel(DevState st, Dims dm, int seq, int prefill, int policy) {
  if (threadIdx.x == 0) {
    st.n_cache[seq] = 0;
    st.n_seen[seq] = 0;
    st.prefill[seq] = prefill;
    st.policy[seq] = policy;
    st.hp_parity[seq] = 0;
    st.first_changed[seq] = 0;
    st.ticket[seq] = 0u;
    st.n_kept[seq] = 0;
  }
  if (dm.layer_budgets)
    for (int l = threadIdx.x; l < dm.L; l += blockDim.x) {
      st.n_layer[seq * dm.L + l] = 0;
      st.lfirst[seq * dm.L + l] = 0;
    }
}

cudaError_t launch_init_state(const DevState& st, const Dims& dm, cudaStream_t stream) {
  init_state_kernel<<<(dm.S + 255) / 256, 256, 0, stream>>>(st, dm);
  return cudaGetLastError();
}

cudaError_t launch_reset_seq(const DevState& st, const Dims& dm, int seq, int prefill, int policy,
                             cudaStream_t stream) {
  reset_seq_kernel<<<1, 32, 0, stream>>>(st, dm, seq, prefill, policy);
  return cudaGetLastError();
}

}  // namespace epikv
