// k_paper.cu -- CUDA-core kernels of the paper's own environment (paper
// §IV-B; device code in paper_device.cuh): reset, action replay,
// observation, and the fused rollout with fp32 networks.  One thread per env;
// the env's dynamic state stays in registers across the T steps, the action
// history in its state rows.
#include "auv_kernels.h"
#include "mlp_fp32.cuh"
#include "paper_device.cuh"

namespace auv {

namespace {

using paper::kAct;
using paper::kObs;

__global__ void __launch_bounds__(256) k_paper_reset(const Model M, Buffers B,
                                                     const uint8_t* __restrict__ mask) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  if (mask && !mask[i]) return;
  paper::Env e;
  e.ep = B.episode[i];
  paper::reset_env(M, M.id_base + (uint32_t)i, e, paper::hist_rows(B.state, M.n, i));
  paper::store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
}

constexpr int kReplayThreads = 128;

__global__ void __launch_bounds__(kReplayThreads, 4) k_paper_replay(const Model M, Buffers B,
                                                      const float* __restrict__ act, int T,
                                                      float* __restrict__ rew,
                                                      uint8_t* __restrict__ done, float* trace,
                                                      Status* st) {
  // The action history lives in shared memory for the whole launch (one
  // column per thread, copied in and out once): its reads every step are
  // shared-memory loads instead of L2 round trips.
  __shared__ float hist[6 * paper::kHist * kReplayThreads];
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  const paper::HistS h{hist + threadIdx.x, kReplayThreads};
  for (int r = 0; r < 6 * paper::kHist; ++r) h.st(r, B.state[(13 + r) * n + i]);
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  bool bad = false;
  // Step t + 1's actions are loaded while step t integrates, so their DRAM
  // latency is hidden behind a step of arithmetic.
  float a_next[kAct];
#pragma unroll
  for (int k = 0; k < kAct; ++k) a_next[k] = T > 0 ? __ldg(act + (size_t)k * n + i) : 0.0f;
  for (int t = 0; t < T; ++t) {
    float a[kAct];
#pragma unroll
    for (int k = 0; k < kAct; ++k) a[k] = a_next[k];
    if (t + 1 < T) {
#pragma unroll
      for (int k = 0; k < kAct; ++k)
        a_next[k] = __ldg(act + ((size_t)(t + 1) * kAct + k) * n + i);
    }
    bool d;
    const float r = paper::physics_step(M, M.id_base + (uint32_t)i, e, a, h, &d);
    rew[(size_t)t * n + i] = r;
    done[(size_t)t * n + i] = d ? 1 : 0;
    if (trace) paper::trace_state(M, h, trace + (size_t)t * paper::kStateF * n, i, e);
    bad |= !paper::env_finite(e);
  }
  if (bad) flag_nan(st, i);
  paper::store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  for (int r = 0; r < 6 * paper::kHist; ++r) B.state[(13 + r) * n + i] = h.ld(r);
}

__global__ void __launch_bounds__(256) k_paper_observe(const Model M, Buffers B,
                                                       float* __restrict__ obs) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  float o[kObs];
  paper::observe(e, o);
#pragma unroll
  for (int k = 0; k < kObs; ++k) obs[(size_t)k * M.n + i] = o[k];
}

// Gaussian head over the wrench: the first six of the step's eight normals.
__device__ __forceinline__ void sample_wrench(const Model& M, uint32_t id, uint64_t t_g,
                                              const float* head, float a[kAct], float* logp) {
  float eps[8];
  action_noise(id, M.seed, t_g, eps);
  float lp = 0.0f;
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    float ls = M.logstd_fixed[k];
    if (M.policy_out == 2 * kAct) ls = fminf(fmaxf(head[kAct + k], M.logstd_min), M.logstd_max);
    a[k] = fmaf(expf(ls), eps[k], head[k]);
    lp += -0.5f * eps[k] * eps[k] - ls;
  }
  *logp = lp - (float)kAct * 0.91893853320467274f;
}

template <int H, int OUT>
__global__ void __launch_bounds__(kTile) k_paper_rollout_fp32(const Model M, Buffers B,
                                                              const float* __restrict__ wp,
                                                              const float* __restrict__ wv,
                                                              Traj tr, int T, uint64_t t_g0,
                                                              Status* st) {
  extern __shared__ float hs_all[];
  const int i = blockIdx.x * kTile + threadIdx.x;
  if (i >= M.n) return;
  float* hs = hs_all + threadIdx.x;
  const size_t n = (size_t)M.n;
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  bool bad = false;
  for (int t = 0; t < T; ++t) {
    float o[kObs];
    paper::observe(e, o);
    float head[OUT];
    mlp_fp32<kObs, H, OUT>(wp, o, hs, head);
    float a[kAct], lp;
    sample_wrench(M, M.id_base + (uint32_t)i, t_g0 + (uint64_t)t, head, a, &lp);
    if (tr.value) {
      float v[1];
      mlp_fp32<kObs, H, 1>(wv, o, hs, v);
      tr.value[(size_t)t * n + i] = v[0];
    }
    if (tr.obs) {
#pragma unroll
      for (int k = 0; k < kObs; ++k) tr.obs[((size_t)t * kObs + k) * n + i] = o[k];
    }
    if (tr.act) {
#pragma unroll
      for (int k = 0; k < kAct; ++k) tr.act[((size_t)t * kAct + k) * n + i] = a[k];
    }
    if (tr.logp) tr.logp[(size_t)t * n + i] = lp;
    bool d;
    const float r = paper::physics_step(M, M.id_base + (uint32_t)i, e, a,
                                        paper::hist_rows(B.state, M.n, i), &d);
    if (tr.rew) tr.rew[(size_t)t * n + i] = r;
    if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
    bad |= !paper::env_finite(e);
  }
  if (bad) flag_nan(st, i);
  paper::store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
}

inline int blocks_for(int n, int b) { return (n + b - 1) / b; }

template <int H, int OUT>
cudaError_t paper_rollout_fp32_impl(const Model& M, const Buffers& B, const float* wp,
                                    const float* wv, const Traj& tr, int T, uint64_t t_g0,
                                    Status* st, cudaStream_t s) {
  const size_t smem = (size_t)H * kTile * sizeof(float);
  cudaError_t err = cudaFuncSetAttribute(k_paper_rollout_fp32<H, OUT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  k_paper_rollout_fp32<H, OUT><<<blocks_for(M.n, kTile), kTile, smem, s>>>(M, B, wp, wv, tr, T,
                                                                          t_g0, st);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_paper_reset(const Model& M, const Buffers& B, const uint8_t* mask,
                               cudaStream_t s) {
  k_paper_reset<<<blocks_for(M.n, 256), 256, 0, s>>>(M, B, mask);
  return cudaGetLastError();
}

cudaError_t launch_paper_replay(const Model& M, const Buffers& B, const float* act, int T,
                                float* rew, uint8_t* done, float* trace, Status* st,
                                cudaStream_t s) {
  k_paper_replay<<<blocks_for(M.n, kReplayThreads), kReplayThreads, 0, s>>>(M, B, act, T, rew,
                                                                             done, trace, st);
  return cudaGetLastError();
}

cudaError_t launch_paper_observe(const Model& M, const Buffers& B, float* obs, cudaStream_t s) {
  k_paper_observe<<<blocks_for(M.n, 256), 256, 0, s>>>(M, B, obs);
  return cudaGetLastError();
}

cudaError_t launch_paper_rollout_fp32(const Model& M, const Buffers& B, const float* wp,
                                      const float* wv, const Traj& tr, int T, uint64_t t_g0,
                                      Status* st, cudaStream_t s) {
  const int H = M.hidden, O = M.policy_out;
  if (H == 64 && O == 6) return paper_rollout_fp32_impl<64, 6>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (H == 64 && O == 12) return paper_rollout_fp32_impl<64, 12>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (H == 256 && O == 6) return paper_rollout_fp32_impl<256, 6>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (H == 256 && O == 12) return paper_rollout_fp32_impl<256, 12>(M, B, wp, wv, tr, T, t_g0, st, s);
  return cudaErrorInvalidValue;
}

}  // namespace auv
