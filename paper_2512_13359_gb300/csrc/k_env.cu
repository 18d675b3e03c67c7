// k_env.cu -- CUDA-core kernels of the batched AUV rollout: episode reset,
// action replay, observation, raw Philox words, and the fp32 rollout whose
// policy/value networks run on the FP32 pipe (the exact-arithmetic mode).
// One thread owns one environment for the whole launch; its state lives in
// registers across all T control steps and touches HBM only at the start and
// the end (plus the trajectory rows it writes).
#include "auv_kernels.h"
#include "mlp_fp32.cuh"

namespace auv {

// ---------------------------------------------------------------------------
// Reset: env i starts a new episode if mask == NULL or mask[i] != 0.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_reset(const Model M, Buffers B, const uint8_t* mask) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  if (mask && !mask[i]) return;
  Env e;
  e.ep = B.episode[i];
  reset_env(M, M.id_base + (uint32_t)i, e);
  store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
}

// ---------------------------------------------------------------------------
// Action replay: T control steps with given actions act[T][8][N].
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(128, 4) k_replay(const Model M, Buffers B,
                                                const float* __restrict__ act, int T,
                                                float* __restrict__ rew, uint8_t* __restrict__ done,
                                                float* __restrict__ trace, Status* st) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
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
    const float r = physics_step(M, M.id_base + (uint32_t)i, e, a, &d);
    rew[(size_t)t * n + i] = r;
    done[(size_t)t * n + i] = d ? 1 : 0;
    if (trace) store_state(M, trace + (size_t)t * kStateF * n, i, e);
    bad |= !env_finite(e);
  }
  if (bad) flag_nan(st, i);
  store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
}

__global__ void __launch_bounds__(256) k_observe(const Model M, Buffers B, float* __restrict__ obs) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  float o[kObs];
  observe(e, o);
#pragma unroll
  for (int k = 0; k < kObs; ++k) obs[(size_t)k * M.n + i] = o[k];
}

__global__ void __launch_bounds__(256) k_draw_words(const Model M, uint32_t stream_id,
                                                    uint64_t index, int n_blocks,
                                                    uint32_t* __restrict__ out) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  for (int b = 0; b < n_blocks; ++b) {
    const uint4 r = philox10((uint32_t)index, (uint32_t)(index >> 32), stream_id, (uint32_t)b,
                             M.id_base + (uint32_t)i, M.seed);
    out[(size_t)(4 * b + 0) * n + i] = r.x;
    out[(size_t)(4 * b + 1) * n + i] = r.y;
    out[(size_t)(4 * b + 2) * n + i] = r.z;
    out[(size_t)(4 * b + 3) * n + i] = r.w;
  }
}

// Gaussian head: mean, log-std (fixed or clamped head), sampled action and
// its log-density from the env's action-noise normals.
__device__ __forceinline__ void sample_action(const Model& M, uint32_t id, uint64_t t_g,
                                              const float* head, float a[kAct], float* logp) {
  float eps[kAct];
  action_noise(id, M.seed, t_g, eps);
  float lp = 0.0f;
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    float ls = M.logstd_fixed[k];
    if (M.policy_out == 16) ls = fminf(fmaxf(head[kAct + k], M.logstd_min), M.logstd_max);
    a[k] = fmaf(expf(ls), eps[k], head[k]);
    lp += -0.5f * eps[k] * eps[k] - ls;
  }
  *logp = lp - (float)kAct * 0.91893853320467274f;
}

template <int H, int OUT>
__global__ void __launch_bounds__(kTile) k_rollout_fp32(const Model M, Buffers B,
                                                        const float* __restrict__ wp,
                                                        const float* __restrict__ wv, Traj tr,
                                                        int T, uint64_t t_g0, Status* st) {
  extern __shared__ float hs_all[];
  const int i = blockIdx.x * kTile + threadIdx.x;
  if (i >= M.n) return;
  float* hs = hs_all + threadIdx.x;
  const size_t n = (size_t)M.n;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  bool bad = false;
  for (int t = 0; t < T; ++t) {
    float o[kObs];
    observe(e, o);
    float head[OUT];
    mlp_fp32<kObs, H, OUT>(wp, o, hs, head);
    float a[kAct], lp;
    sample_action(M, M.id_base + (uint32_t)i, t_g0 + (uint64_t)t, head, a, &lp);
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
    const float r = physics_step(M, M.id_base + (uint32_t)i, e, a, &d);
    if (tr.rew) tr.rew[(size_t)t * n + i] = r;
    if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
    bad |= !env_finite(e);
  }
  if (bad) flag_nan(st, i);
  store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
}

// Small batches (tens to a few thousand envs): the one-thread-per-env kernel
// above leaves each env's network as one thread's serial chain on a handful
// of SMs.  Here a team of H threads evaluates each env's networks, thread j
// computing hidden unit j of both layers and output j of the head, each sum
// in mlp_fp32's order (the same floats); the team's first thread holds the
// env's state and runs the sampling and the physics.  H = 64, four envs per
// 256-thread CTA.
template <int H, int OUT>
__global__ void __launch_bounds__(256) k_rollout_fp32_team(const Model M, Buffers B,
                                                           const float* __restrict__ wp,
                                                           const float* __restrict__ wv, Traj tr,
                                                           int T, uint64_t t_g0, Status* st) {
  static_assert(H >= OUT && 256 % H == 0, "team shape");
  constexpr int E = 256 / H;
  __shared__ float s_x[E][kObs];
  __shared__ float s_h1[E][H];
  __shared__ float s_h2[E][H];
  __shared__ float s_out[E][OUT + 1];   // policy head, then the value
  const int el = threadIdx.x / H, j = threadIdx.x % H;
  const int i = blockIdx.x * E + el;
  const bool active = i < M.n, lead = j == 0;
  const size_t n = (size_t)M.n;
  // hidden unit j of layer 1 / layer 2 and output o of the head of one
  // network (row-major weights, mlp_fp32's layout and summation order)
  auto unit1 = [&](const float* w, int u) {
    const float* W1 = w;
    const float* b1 = W1 + H * kObs;
    float s = __ldg(b1 + u);
    const float2* row = reinterpret_cast<const float2*>(W1 + u * kObs);
#pragma unroll
    for (int i2 = 0; i2 < kObs / 2; ++i2) {
      const float2 wv2 = __ldg(row + i2);
      s = fmaf(wv2.x, s_x[el][2 * i2], s);
      s = fmaf(wv2.y, s_x[el][2 * i2 + 1], s);
    }
    s_h1[el][u] = tanhf(s);
  };
  auto unit2 = [&](const float* w, int u) {
    const float* W2 = w + H * kObs + H;
    const float* b2 = W2 + H * H;
    float s0 = __ldg(b2 + u), s1 = 0.0f;
    const float4* row = reinterpret_cast<const float4*>(W2 + (size_t)u * H);
#pragma unroll 8
    for (int k4 = 0; k4 < H / 4; ++k4) {
      const float4 q = __ldg(row + k4);
      s0 = fmaf(q.x, s_h1[el][4 * k4 + 0], s0);
      s1 = fmaf(q.y, s_h1[el][4 * k4 + 1], s1);
      s0 = fmaf(q.z, s_h1[el][4 * k4 + 2], s0);
      s1 = fmaf(q.w, s_h1[el][4 * k4 + 3], s1);
    }
    s_h2[el][u] = tanhf(s0 + s1);
  };
  auto head = [&](const float* w, int out_dim, int o) {
    const float* W3 = w + H * kObs + H + H * H + H;
    const float* b3 = W3 + out_dim * H;
    float s = __ldg(b3 + o);
    for (int u = 0; u < H; ++u) s = fmaf(__ldg(W3 + o * H + u), s_h2[el][u], s);
    return s;
  };
  Env e;
  if (lead && active) load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  bool bad = false;
  for (int t = 0; t < T; ++t) {
    if (lead) {
      float o[kObs];
      if (active) {
        observe(e, o);
        if (tr.obs) {
#pragma unroll
          for (int k = 0; k < kObs; ++k) tr.obs[((size_t)t * kObs + k) * n + i] = o[k];
        }
      } else {
#pragma unroll
        for (int k = 0; k < kObs; ++k) o[k] = 0.0f;
      }
#pragma unroll
      for (int k = 0; k < kObs; ++k) s_x[el][k] = o[k];
    }
    __syncthreads();
    unit1(wp, j);
    __syncthreads();
    unit2(wp, j);
    __syncthreads();
    if (j < OUT) s_out[el][j] = head(wp, OUT, j);
    if (tr.value) unit1(wv, j);       // the value network's layer 1 (s_h1 is free)
    __syncthreads();
    if (tr.value) {
      unit2(wv, j);
      __syncthreads();
      if (j == 0) s_out[el][OUT] = head(wv, 1, 0);
      __syncthreads();
    }
    if (lead && active) {
      float hd[OUT];
#pragma unroll
      for (int k = 0; k < OUT; ++k) hd[k] = s_out[el][k];
      float a[kAct], lp;
      sample_action(M, M.id_base + (uint32_t)i, t_g0 + (uint64_t)t, hd, a, &lp);
      if (tr.value) tr.value[(size_t)t * n + i] = s_out[el][OUT];
      if (tr.act) {
#pragma unroll
        for (int k = 0; k < kAct; ++k) tr.act[((size_t)t * kAct + k) * n + i] = a[k];
      }
      if (tr.logp) tr.logp[(size_t)t * n + i] = lp;
      bool d;
      const float r = physics_step(M, M.id_base + (uint32_t)i, e, a, &d);
      if (tr.rew) tr.rew[(size_t)t * n + i] = r;
      if (tr.done) tr.done[(size_t)t * n + i] = d ? 1 : 0;
      bad |= !env_finite(e);
    }
  }
  if (lead && active) {
    if (bad) flag_nan(st, i);
    store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  }
}

template <int IN, int H, int OUT>
__global__ void __launch_bounds__(kTile) k_forward_fp32(const float* __restrict__ wp,
                                                        const float* __restrict__ wv,
                                                        const float* __restrict__ obs, int n,
                                                        float* __restrict__ head,
                                                        float* __restrict__ value) {
  extern __shared__ float hs_all[];
  const int i = blockIdx.x * kTile + threadIdx.x;
  if (i >= n) return;
  float* hs = hs_all + threadIdx.x;
  float o[IN];
#pragma unroll
  for (int k = 0; k < IN; ++k) o[k] = obs[(size_t)i * IN + k];
  float h[OUT];
  mlp_fp32<IN, H, OUT>(wp, o, hs, h);
#pragma unroll
  for (int k = 0; k < OUT; ++k) head[(size_t)i * OUT + k] = h[k];
  if (value) {
    float v[1];
    mlp_fp32<IN, H, 1>(wv, o, hs, v);
    value[i] = v[0];
  }
}

// Value network on trajectory-layout observations: row r = t*n + i reads
// obs[(t*IN + k)*n + i].
template <int IN, int H>
__global__ void __launch_bounds__(kTile) k_value_fp32(const float* __restrict__ wv,
                                                      const float* __restrict__ obs, size_t rows,
                                                      int n, float* __restrict__ value) {
  extern __shared__ float hs_all[];
  const size_t r = (size_t)blockIdx.x * kTile + threadIdx.x;
  if (r >= rows) return;
  float* hs = hs_all + threadIdx.x;
  const size_t t = r / (size_t)n, i = r % (size_t)n;
  float o[IN];
#pragma unroll
  for (int k = 0; k < IN; ++k) o[k] = obs[(t * IN + k) * n + i];
  float v[1];
  mlp_fp32<IN, H, 1>(wv, o, hs, v);
  value[r] = v[0];
}

// ---------------------------------------------------------------------------
// Host-side launchers (called from the C ABI layer).
// ---------------------------------------------------------------------------
static inline int blocks_for(int n, int b) { return (n + b - 1) / b; }

cudaError_t launch_reset(const Model& M, const Buffers& B, const uint8_t* mask, cudaStream_t s) {
  k_reset<<<blocks_for(M.n, 256), 256, 0, s>>>(M, B, mask);
  return cudaGetLastError();
}

cudaError_t launch_replay(const Model& M, const Buffers& B, const float* act, int T, float* rew,
                          uint8_t* done, float* trace, Status* st, cudaStream_t s) {
  k_replay<<<blocks_for(M.n, 128), 128, 0, s>>>(M, B, act, T, rew, done, trace, st);
  return cudaGetLastError();
}

cudaError_t launch_observe(const Model& M, const Buffers& B, float* obs, cudaStream_t s) {
  k_observe<<<blocks_for(M.n, 256), 256, 0, s>>>(M, B, obs);
  return cudaGetLastError();
}

cudaError_t launch_draw_words(const Model& M, uint32_t stream_id, uint64_t index, int n_blocks,
                              uint32_t* out, cudaStream_t s) {
  k_draw_words<<<blocks_for(M.n, 256), 256, 0, s>>>(M, stream_id, index, n_blocks, out);
  return cudaGetLastError();
}

// Batches at most this large run the team kernel (hidden width 64).
constexpr int kTeamMaxEnvs = 2048;

template <int H, int OUT>
static cudaError_t rollout_fp32_impl(const Model& M, const Buffers& B, const float* wp,
                                     const float* wv, const Traj& tr, int T, uint64_t t_g0,
                                     Status* st, cudaStream_t s) {
  if constexpr (H == 64) {
    if (M.n <= kTeamMaxEnvs) {
      k_rollout_fp32_team<H, OUT><<<blocks_for(M.n, 256 / H), 256, 0, s>>>(M, B, wp, wv, tr, T,
                                                                           t_g0, st);
      return cudaGetLastError();
    }
  }
  const size_t smem = (size_t)H * kTile * sizeof(float);
  cudaError_t err = cudaFuncSetAttribute(k_rollout_fp32<H, OUT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  k_rollout_fp32<H, OUT><<<blocks_for(M.n, kTile), kTile, smem, s>>>(M, B, wp, wv, tr, T, t_g0, st);
  return cudaGetLastError();
}

cudaError_t launch_rollout_fp32(const Model& M, const Buffers& B, const float* wp,
                                const float* wv, const Traj& tr, int T, uint64_t t_g0, Status* st,
                                cudaStream_t s) {
  if (M.hidden == 64 && M.policy_out == 8) return rollout_fp32_impl<64, 8>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (M.hidden == 64 && M.policy_out == 16) return rollout_fp32_impl<64, 16>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (M.hidden == 256 && M.policy_out == 8) return rollout_fp32_impl<256, 8>(M, B, wp, wv, tr, T, t_g0, st, s);
  if (M.hidden == 256 && M.policy_out == 16) return rollout_fp32_impl<256, 16>(M, B, wp, wv, tr, T, t_g0, st, s);
  return cudaErrorInvalidValue;
}

template <int IN, int H>
static cudaError_t value_fp32_impl(const float* wv, const float* obs, size_t rows, int n,
                                   float* value, cudaStream_t s) {
  const size_t smem = (size_t)H * kTile * sizeof(float);
  cudaError_t err = cudaFuncSetAttribute(k_value_fp32<IN, H>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  const size_t blocks = (rows + kTile - 1) / kTile;
  k_value_fp32<IN, H><<<(unsigned)blocks, kTile, smem, s>>>(wv, obs, rows, n, value);
  return cudaGetLastError();
}

cudaError_t launch_value_fp32(const Model& M, const float* wv, const float* obs, size_t rows,
                              int n, float* value, cudaStream_t s) {
  const bool paper = M.model == 1;
  if (M.hidden == 64)
    return paper ? value_fp32_impl<12, 64>(wv, obs, rows, n, value, s)
                 : value_fp32_impl<kObs, 64>(wv, obs, rows, n, value, s);
  if (M.hidden == 256)
    return paper ? value_fp32_impl<12, 256>(wv, obs, rows, n, value, s)
                 : value_fp32_impl<kObs, 256>(wv, obs, rows, n, value, s);
  return cudaErrorInvalidValue;
}

template <int IN, int H, int OUT>
static cudaError_t forward_fp32_impl(const float* wp, const float* wv, const float* obs, int n,
                                     float* head, float* value, cudaStream_t s) {
  const size_t smem = (size_t)H * kTile * sizeof(float);
  cudaError_t err = cudaFuncSetAttribute(k_forward_fp32<IN, H, OUT>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (err != cudaSuccess) return err;
  k_forward_fp32<IN, H, OUT><<<blocks_for(n, kTile), kTile, smem, s>>>(wp, wv, obs, n, head,
                                                                        value);
  return cudaGetLastError();
}

cudaError_t launch_forward_fp32(const Model& M, const float* wp, const float* wv,
                                const float* obs, int n, float* head, float* value,
                                cudaStream_t s) {
  const int H = M.hidden, O = M.policy_out;
  if (M.model == 1) {
    if (H == 64 && O == 6) return forward_fp32_impl<12, 64, 6>(wp, wv, obs, n, head, value, s);
    if (H == 64 && O == 12) return forward_fp32_impl<12, 64, 12>(wp, wv, obs, n, head, value, s);
    if (H == 256 && O == 6) return forward_fp32_impl<12, 256, 6>(wp, wv, obs, n, head, value, s);
    if (H == 256 && O == 12) return forward_fp32_impl<12, 256, 12>(wp, wv, obs, n, head, value, s);
    return cudaErrorInvalidValue;
  }
  if (H == 64 && O == 8) return forward_fp32_impl<kObs, 64, 8>(wp, wv, obs, n, head, value, s);
  if (H == 64 && O == 16) return forward_fp32_impl<kObs, 64, 16>(wp, wv, obs, n, head, value, s);
  if (H == 256 && O == 8) return forward_fp32_impl<kObs, 256, 8>(wp, wv, obs, n, head, value, s);
  if (H == 256 && O == 16) return forward_fp32_impl<kObs, 256, 16>(wp, wv, obs, n, head, value, s);
  return cudaErrorInvalidValue;
}

}  // namespace auv
