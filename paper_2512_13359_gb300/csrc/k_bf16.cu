// k_bf16.cu -- tensor-core network path (placeholder until the tcgen05
// kernels land: every entry reports "not supported").
#include "auv_bf16.h"

namespace auv {

size_t bf16_policy_image_bytes() { return 1024; }
size_t bf16_value_image_bytes() { return 1024; }

cudaError_t launch_pack_bf16(const Model&, const float*, const float*, void*, void*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t launch_rollout_bf16(const Model&, const Buffers&, const void*, const Traj&, int,
                                uint64_t, Status*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t launch_value_bf16(const Model&, const void*, const float*, const float*, size_t, int,
                              float*, Status*, cudaStream_t) {
  return cudaErrorNotSupported;
}
cudaError_t launch_forward_bf16(const Model&, const void*, const void*, const float*,
                                const float*, int, float*, float*, Status*, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace auv
