// k_ppo.cu -- on-GPU pieces of the PPO learner that consume the rollout's
// SoA trajectory (paper §III-A: PPO, Schulman et al. 2017).
//
// Generalised advantage estimation (Schulman et al. 2016) over [T][N]
// arrays, one thread per env walking t = T-1 .. 0:
//   delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,   V_T = last_value
//   A_t = delta_t + gamma lambda (1 - d_t) A_{t+1};  R_t = A_t + V_t.
// The kernel is bound by HBM: 17 bytes per env-step (reward, done, value in;
// advantage, return out).  Each thread loads a block of kU steps before it
// runs their recursion, so that every warp keeps 3 kU coalesced loads in
// flight (16-step blocks: 3.1 TB/s at 65,536 envs x 128 steps, 4.3 TB/s at
// 262,144; 8- and 32-step blocks measured slower).
#include "auv_kernels.h"

namespace auv {

namespace {

constexpr int kU = 16;

__global__ void __launch_bounds__(256) k_gae(int n, int T, const float* __restrict__ rew,
                                             const uint8_t* __restrict__ done,
                                             const float* __restrict__ value,
                                             const float* __restrict__ last_value, float gamma,
                                             float gl, float* __restrict__ adv,
                                             float* __restrict__ ret) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n) return;
  const size_t N = (size_t)n;
  float a_next = 0.0f;
  float v_next = __ldg(last_value + i);
  for (int hi = T; hi > 0; hi -= kU) {
    const int cnt = hi < kU ? hi : kU;
    const int lo = hi - cnt;
    float r[kU], v[kU], nt[kU];
#pragma unroll
    for (int k = 0; k < kU; ++k) {
      if (k < cnt) {
        const size_t o = (size_t)(lo + k) * N + i;
        r[k] = __ldg(rew + o);
        v[k] = __ldg(value + o);
        nt[k] = __ldg(done + o) ? 0.0f : 1.0f;
      }
    }
#pragma unroll
    for (int k = kU - 1; k >= 0; --k) {
      if (k < cnt) {
        const float delta = fmaf(gamma * nt[k], v_next, r[k]) - v[k];
        a_next = fmaf(gl * nt[k], a_next, delta);
        const size_t o = (size_t)(lo + k) * N + i;
        adv[o] = a_next;
        ret[o] = a_next + v[k];
        v_next = v[k];
      }
    }
  }
}

}  // namespace

cudaError_t launch_gae(int n, int T, const float* rew, const uint8_t* done, const float* value,
                       const float* last_value, float gamma, float lam, float* adv, float* ret,
                       cudaStream_t s) {
  k_gae<<<(n + 255) / 256, 256, 0, s>>>(n, T, rew, done, value, last_value, gamma, gamma * lam,
                                        adv, ret);
  return cudaGetLastError();
}

}  // namespace auv
