// auv_bf16.h -- internal interface of the tensor-core (tcgen05, bf16 operands,
// fp32 accumulation in tensor memory) network path.
#pragma once

#include "auv_kernels.h"

namespace auv {

// Bytes of the packed operand images the bf16 kernels stream into shared
// memory (policy and value networks, hidden width 256).
size_t bf16_policy_image_bytes();
size_t bf16_value_image_bytes();

// fp32 row-major weights -> packed bf16 images (round to nearest even).
cudaError_t launch_pack_bf16(const Model& M, const float* wp_f32, const float* wv_f32,
                             void* wp_packed, void* wv_packed, cudaStream_t s);

// The same from explicit widths: network input in_dim (<= 18), policy head
// policy_out (<= 16); either weight pointer may be NULL.
cudaError_t launch_pack_bf16_dims(int in_dim, int policy_out, const float* wp_f32,
                                  const float* wv_f32, void* wp_packed, void* wv_packed,
                                  cudaStream_t s);

// Learner forward of one network (policy: out_dim <= 16 head outputs; value:
// one) on `rows` bf16 input rows x[r][ldx] (ldx a multiple of 8, > in_dim):
// the bf16 hidden activations to h1, h2 ([rows][ldh], columns 0..255; ldh a
// multiple of 8) and the head to out[r][ldo], fp32.
cudaError_t launch_learn_forward_bf16(bool policy, const void* packed, int in_dim, int out_dim,
                                      const uint16_t* x, int ldx, size_t rows, uint16_t* h1,
                                      uint16_t* h2, int ldh, float* out, int ldo, Status* st,
                                      cudaStream_t s);

// Learner backward-data of one network on the same engine, from the packed
// transposed weights (launch_pack_back_bf16: W3^T and W2^T of the flat fp32
// weights; in_dim the network input width, out_dim its head width <= 16):
// gz2 = (W3^T gy) (1 - h2^2) and gz1 = (W2^T gz2) (1 - h1^2), bf16, for
// `rows` rows (gy [rows][ldy], h1, h2 [rows][ldh], gz2 [rows][ldz2],
// gz1 [rows][ldz1]; strides multiples of 8, ldy >= 8 ceil(out_dim / 8)).
// gz1 may be h2 itself: each row is read before it is written, by one thread.
size_t bf16_back_image_bytes();
cudaError_t launch_pack_back_bf16(int in_dim, int out_dim, const float* w_f32, void* packed,
                                  cudaStream_t s);
// The learner's forward and backward images of both networks in one launch
// (launch_pack_bf16_dims and launch_pack_back_bf16 of each; a NULL weight
// pointer skips that network's two images).
cudaError_t launch_pack_learner_bf16(int in_dim, int policy_out, const float* wp_f32,
                                     const float* wv_f32, void* wp_packed, void* wv_packed,
                                     void* bp_packed, void* bv_packed, cudaStream_t s);
cudaError_t launch_learn_backward_bf16(const void* packed, int out_dim, const uint16_t* gy, int ldy,
                                       size_t rows, const uint16_t* h2, const uint16_t* h1, int ldh,
                                       uint16_t* gz2, int ldz2, uint16_t* gz1, int ldz1, Status* st,
                                       cudaStream_t s);

// Fused rollout with the policy network on tcgen05.
// tf32 tensor-core rollout (k_tf32.cu): Fossen model, hidden 256, policy head
// 8 or 16, no value network; packed image from the fp32 policy weights.
size_t tf32_policy_image_bytes();
cudaError_t launch_pack_tf32(const Model& M, const float* wp_f32, void* packed, cudaStream_t s);
cudaError_t launch_rollout_tf32(const Model& M, const Buffers& B, const void* packed,
                                const Traj& tr, int T, uint64_t t_g0, Status* st, cudaStream_t s);

cudaError_t launch_rollout_bf16(const Model& M, const Buffers& B, const void* wp_packed,
                                const Traj& tr, int T, uint64_t t_g0, Status* st, cudaStream_t s);

// Value network over `rows` stored observations obs[t][18][n] (row r = t*n + i).
cudaError_t launch_value_bf16(const Model& M, const void* wv_packed, const float* wv_f32,
                              const float* obs, size_t rows, int n, float* value, Status* st,
                              cudaStream_t s);

// Networks on caller observations obs[n][18] (row-major).
cudaError_t launch_forward_bf16(const Model& M, const void* wp_packed, const void* wv_packed,
                                const float* wv_f32, const float* obs, int n, float* head,
                                float* value, Status* st, cudaStream_t s);

// SM count of the current device (looked up once per device).
int engine_sm_count();

// Failure-detection self-test (a bounded wait that is made to run out).
cudaError_t launch_wait_selftest(Status* st, uint64_t limit_ns, cudaStream_t s);

}  // namespace auv
