// paper_device.cuh -- device code of the paper's own environment (paper
// §IV-B "Environment Specifications", Eqs. (1)-(7), §IV-C), next to the
// thruster-level Fossen model of auv_device.cuh:
//  - action: a normalised body wrench a = [F; tau] in [-1, 1]^6, clipped and
//    scaled by F_max and tau_max (Eq. 1);
//  - dynamics: a free rigid body (no added mass) in still water under the
//    inertia fluid model: quadratic drag -kf_i |v_i| v_i and -kt_i |w_i| w_i
//    of the uniform box with the body's mass and inertia, Stokes resistance
//    -c_visc_f v and -c_visc_t w, and buoyancy folded into an effective
//    gravity (0, 0, -g) at the centre of mass, g redrawn per episode (§IV-C);
//    the semi-implicit Euler substep and exponential-map attitude update of
//    the Fossen model;
//  - observation (12): R^T (p - p_d), the axis-angle vector of
//    conj(q_d) (x) q on the short way round, v, w (§IV-B1);
//  - reward: -w_pos |D dp_b|^2 - w_att |theta_e|^2 - w_act |a_c(3:6)|^2
//    - w_vel |w|^2 - w_mavg |a_c - mean of the K previous a_c|^2 (Eqs. 2-7).
// The K-slot history of clipped actions lives in state rows 13.. (slot j,
// component k at row 13 + 6 j + k); it is read and written in global memory
// every step, not held in registers.
#pragma once

#include "auv_device.cuh"

namespace auv {
namespace paper {

constexpr int kObs = 12;
constexpr int kAct = 6;
constexpr int kHist = 8;
constexpr int kStateF = 13 + 6 * kHist;
constexpr int kParamF = 8;

struct Env {
  float p[3], q[4], nu[6];
  float pd[3], qd[4], g;
  int t_ep;
  uint32_t ep;
};

// The K-slot action history of one env, entry r = 6 j + k (slot j,
// component k).  HistG: the state rows 13.. of [kStateF][n] in global memory,
// read past L1; HistS: a copy in shared memory, one column per thread.
struct HistG {
  float* p;
  int s;   // r * s < 48 n fits an int for every env count the state array allows
  __device__ __forceinline__ float ld(int r) const { return __ldcg(p + r * s); }
  __device__ __forceinline__ void st(int r, float v) const { p[r * s] = v; }
};
struct HistS {
  float* p;
  int s;
  __device__ __forceinline__ float ld(int r) const { return p[r * s]; }
  __device__ __forceinline__ void st(int r, float v) const { p[r * s] = v; }
};
__device__ __forceinline__ HistG hist_rows(float* st, int n, int i) {
  return HistG{st + 13 * (size_t)n + i, n};
}

__device__ __forceinline__ void load_env(const Model& M, const float* st, const float* pr,
                                         const int* t_ep, const uint32_t* ep, int i, Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) e.p[k] = st[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.q[k] = st[(3 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nu[k] = st[(7 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.pd[k] = pr[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.qd[k] = pr[(3 + k) * n + i];
  e.g = pr[7 * n + i];
  e.t_ep = t_ep[i];
  e.ep = ep[i];
}

// Rows 0..12 (the history rows are written where they change).
__device__ __forceinline__ void store_state(const Model& M, float* st, int i, const Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) st[k * n + i] = e.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) st[(3 + k) * n + i] = e.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) st[(7 + k) * n + i] = e.nu[k];
}

__device__ __forceinline__ void store_env(const Model& M, float* st, float* pr, int* t_ep,
                                          uint32_t* ep, int i, const Env& e) {
  const int n = M.n;
  store_state(M, st, i, e);
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[k * n + i] = e.pd[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) pr[(3 + k) * n + i] = e.qd[k];
  pr[7 * n + i] = e.g;
  t_ep[i] = e.t_ep;
  ep[i] = e.ep;
}

// Full state of env i to a trace slice (rows 0..12 from registers, the
// history rows copied from the state array).
template <class Hist>
__device__ __forceinline__ void trace_state(const Model& M, const Hist& h, float* tr, int i,
                                            const Env& e) {
  const int n = M.n;
  store_state(M, tr, i, e);
  for (int r = 0; r < 6 * kHist; ++r) tr[(13 + r) * n + i] = h.ld(r);
}

// New episode (counter (episode, 0, 1, block 0..3) of the reset stream):
// goal position, goal roll/pitch/yaw, effective-gravity offset, initial
// position, initial roll/pitch/yaw; velocities and history zeroed.
template <class Hist>
__device__ __forceinline__ void reset_env(const Model& M, uint32_t id, Env& e, const Hist& h) {
  uint32_t w[16];
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const uint4 r = philox10(e.ep, 0u, 1u, (uint32_t)b, id, M.seed);
    w[4 * b + 0] = r.x; w[4 * b + 1] = r.y; w[4 * b + 2] = r.z; w[4 * b + 3] = r.w;
  }
  float u[13];
#pragma unroll
  for (int j = 0; j < 13; ++j) u[j] = uniform01(w[j]);
  euler_quat(sym_draw(u[3], M.goal_att_range), sym_draw(u[4], M.goal_att_range),
             sym_draw(u[5], M.goal_att_range), e.qd);
  euler_quat(sym_draw(u[10], M.init_att_range), sym_draw(u[11], M.init_att_range),
             sym_draw(u[12], M.init_att_range), e.q);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    e.pd[k] = sym_draw(u[k], M.goal_pos_range);
    e.p[k] = sym_draw(u[7 + k], M.init_pos_range);
  }
  e.g = M.dr_enable ? __fadd_rn(M.g_eff0, sym_draw(u[6], M.dr_grav)) : M.g_eff0;
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nu[k] = 0.0f;
  for (int r = 0; r < 6 * kHist; ++r) h.st(r, 0.0f);
  e.t_ep = 0;
  e.ep += 1u;
}

// One substep with the constant wrench tau.
__device__ __forceinline__ void substep(const Model& M, Env& e, const float tau[6]) {
  float R[3][3];
  quat_rot(e.q, R);
  const float v[3] = {e.nu[0], e.nu[1], e.nu[2]};
  const float w[3] = {e.nu[3], e.nu[4], e.nu[5]};
  const float m = M.mass;
  float wxv[3], Iw[3], wxIw[3];
  cross3(w, v, wxv);
#pragma unroll
  for (int k = 0; k < 3; ++k) Iw[k] = M.inertia[k] * w[k];
  cross3(w, Iw, wxIw);
  // effective gravity in the body frame: R^T (0, 0, -m g) = -m g (third row of R)
  const float mg = m * e.g;
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    const float f = -M.kf_drag[k] * fabsf(v[k]) * v[k] - M.c_visc_f * v[k];
    const float t = -M.kt_drag[k] * fabsf(w[k]) * w[k] - M.c_visc_t * w[k];
    const float lin = tau[k] + f - mg * R[2][k] - m * wxv[k];
    const float rot = tau[3 + k] + t - wxIw[k];
    e.nu[k] = fmaf(M.h, lin * M.inv_mass, e.nu[k]);
    e.nu[3 + k] = fmaf(M.h, rot * M.inv_inertia[k], e.nu[3 + k]);
  }
  advance_pose(M.h, R, e.nu, e.p, e.q);
}

// Axis-angle vector of conj(q_d) (x) q with angle in [0, pi].
__device__ __forceinline__ void att_error(const Env& e, float th[3]) {
  const float aw = e.qd[0], ax = -e.qd[1], ay = -e.qd[2], az = -e.qd[3];
  const float bw = e.q[0], bx = e.q[1], by = e.q[2], bz = e.q[3];
  float w = aw * bw - ax * bx - ay * by - az * bz;
  float x = aw * bx + ax * bw + ay * bz - az * by;
  float y = aw * by - ax * bz + ay * bw + az * bx;
  float z = aw * bz + ax * by - ay * bx + az * bw;
  if (w < 0.0f) { w = -w; x = -x; y = -y; z = -z; }
  const float vn = sqrtf(x * x + y * y + z * z);
  const float s = vn > 0.0f ? 2.0f * atan2f(vn, w) / vn : 2.0f / w;
  th[0] = s * x; th[1] = s * y; th[2] = s * z;
}

__device__ __forceinline__ void observe(const Env& e, float o[kObs]) {
  float R[3][3];
  quat_rot(e.q, R);
  const float dp[3] = {e.p[0] - e.pd[0], e.p[1] - e.pd[1], e.p[2] - e.pd[2]};
#pragma unroll
  for (int i = 0; i < 3; ++i) o[i] = R[0][i] * dp[0] + R[1][i] * dp[1] + R[2][i] * dp[2];
  att_error(e, o + 3);
#pragma unroll
  for (int k = 0; k < 6; ++k) o[6 + k] = e.nu[k];
}

// Reward on the post-step state; the history mean is over the K slots as
// they stand before this step's action is entered.
template <class Hist>
__device__ __forceinline__ float reward(const Model& M, const Env& e, const float a_c[kAct],
                                        const Hist& h) {
  float o[kObs];
  observe(e, o);
  float r_pos = 0.0f, r_att = 0.0f, r_act = 0.0f, r_vel = 0.0f;
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    const float d = M.w_axes[k] * o[k];
    r_pos = fmaf(d, d, r_pos);
    r_att = fmaf(o[3 + k], o[3 + k], r_att);
    r_act = fmaf(a_c[3 + k], a_c[3 + k], r_act);
    r_vel = fmaf(e.nu[3 + k], e.nu[3 + k], r_vel);
  }
  const float inv_k = 1.0f / (float)M.mavg_len;
  // Slots in ascending order for each component, as a loop over the
  // compile-time slot count: every slot's loads can be in flight at once.
  float sum[kAct] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int j = 0; j < kHist; ++j) {
    if (j < M.mavg_len) {
#pragma unroll
      for (int k = 0; k < kAct; ++k) sum[k] += h.ld(6 * j + k);
    }
  }
  float r_mavg = 0.0f;
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    const float d = a_c[k] - sum[k] * inv_k;
    r_mavg = fmaf(d, d, r_mavg);
  }
  return -M.w_pos * r_pos - M.w_att * r_att - M.w_act * r_act - M.w_vel * r_vel -
         M.w_mavg * r_mavg;
}

__device__ __forceinline__ bool env_finite(const Env& e) {
  float s = 0.0f;
#pragma unroll
  for (int k = 0; k < 3; ++k) s += e.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) s += e.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) s += e.nu[k];
  return isfinite(s);
}

// One control step with action a: Eq. (1) wrench, substeps, reward, history
// entry (slot t_ep mod K), episode bookkeeping and auto-reset.  st is the
// state array holding this env's history rows.
template <class Hist>
__device__ __forceinline__ float physics_step(const Model& M, uint32_t id, Env& e,
                                              const float a[kAct], const Hist& h, bool* done) {
  float a_c[kAct], tau[6];
#pragma unroll
  for (int k = 0; k < kAct; ++k) a_c[k] = fminf(fmaxf(a[k], -1.0f), 1.0f);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    tau[k] = M.f_max * a_c[k];
    tau[3 + k] = M.tau_max * a_c[3 + k];
  }
  for (int s = 0; s < M.substeps; ++s) substep(M, e, tau);
  const float r = reward(M, e, a_c, h);
  const int slot = e.t_ep % M.mavg_len;
#pragma unroll
  for (int k = 0; k < kAct; ++k) h.st(6 * slot + k, a_c[k]);
  e.t_ep += 1;
  *done = (e.t_ep == M.episode_len);
  if (*done) reset_env(M, id, e, h);
  return r;
}

}  // namespace paper
}  // namespace auv
