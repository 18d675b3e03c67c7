// auv_kernels.h -- internal interface between the C ABI layer (api.cu) and
// the kernel translation units.  Not installed; the public interface is
// include/auvenv.h.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "auv_device.cuh"

namespace auv {

struct Buffers {
  float* state;
  float* params;
  int* t_ep;
  uint32_t* episode;
};

struct Traj {
  float* obs;
  float* act;
  float* logp;
  float* value;
  float* rew;
  uint8_t* done;
};

// CUDA-core kernels (k_env.cu)
cudaError_t launch_reset(const Model& M, const Buffers& B, const uint8_t* mask, cudaStream_t s);
cudaError_t launch_replay(const Model& M, const Buffers& B, const float* act, int T, float* rew,
                          uint8_t* done, float* trace, Status* st, cudaStream_t s);
cudaError_t launch_observe(const Model& M, const Buffers& B, float* obs, cudaStream_t s);
cudaError_t launch_draw_words(const Model& M, uint32_t stream_id, uint64_t index, int n_blocks,
                              uint32_t* out, cudaStream_t s);
cudaError_t launch_rollout_fp32(const Model& M, const Buffers& B, const float* wp,
                                const float* wv, const Traj& tr, int T, uint64_t t_g0, Status* st,
                                cudaStream_t s);
// Value network over stored observations obs[t][obs_dim][n] (row r = t*n + i).
cudaError_t launch_value_fp32(const Model& M, const float* wv, const float* obs, size_t rows,
                              int n, float* value, cudaStream_t s);
cudaError_t launch_forward_fp32(const Model& M, const float* wp, const float* wv,
                                const float* obs, int n, float* head, float* value,
                                cudaStream_t s);

// The paper model's CUDA-core kernels (k_paper.cu)
cudaError_t launch_paper_reset(const Model& M, const Buffers& B, const uint8_t* mask,
                               cudaStream_t s);
cudaError_t launch_paper_replay(const Model& M, const Buffers& B, const float* act, int T,
                                float* rew, uint8_t* done, float* trace, Status* st,
                                cudaStream_t s);
cudaError_t launch_paper_observe(const Model& M, const Buffers& B, float* obs, cudaStream_t s);
cudaError_t launch_paper_rollout_fp32(const Model& M, const Buffers& B, const float* wp,
                                      const float* wv, const Traj& tr, int T, uint64_t t_g0,
                                      Status* st, cudaStream_t s);

// PPO learner pieces (k_ppo.cu)
cudaError_t launch_gae(int n, int T, const float* rew, const uint8_t* done, const float* value,
                       const float* last_value, float gamma, float lam, float* adv, float* ret,
                       cudaStream_t s);

}  // namespace auv
