// auv_device.cuh -- per-environment device arithmetic of the batched AUV
// rollout (arXiv 2512.13359): Philox4x32-10 streams, Box-Muller noise,
// bit-exact episode resets, the Fossen-form 6-DOF substep, observation and
// reward.  Everything here runs on one thread per environment with the state
// held in registers; the kernels in the .cu files compose these pieces.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

namespace auv {

constexpr int kObs = 18;
constexpr int kAct = 8;
constexpr int kStateF = 19;
constexpr int kParamF = 17;

// Model constants, built once on the host from auv_config and passed by value
// as a kernel parameter (constant-bank operands in the generated code).
struct Model {
  int n;              // number of envs
  int substeps;
  int episode_len;
  uint32_t seed;
  uint32_t id_base;   // Philox key word 0 of local env 0
  int dr_enable;
  int policy_out;     // 8 or 16
  int has_value;
  int hidden;
  float h;            // dt / substeps
  float mass;
  float inertia[3];
  float added[6];
  float dlin[6];
  float dquad[6];
  float ghat[3];      // unit gravity direction (world); zero if |g| = 0
  float gnorm;        // |g|
  float alloc_t[48];  // allocation matrix times thrust_max, row-major [6][8]
  float w_pos, w_att, w_act, w_vs;
  float init_pos_range, init_att_range, goal_pos_range, goal_yaw_range, current_range;
  float dr_lo, dr_hi, dr_buoy, dr_cob;
  float logstd_fixed[8];
  float logstd_min, logstd_max;
  // ---- the paper model (model == 1; paper_device.cuh) ----
  int model;          // 0 = Fossen, 1 = paper
  int mavg_len;       // K of Eq. (7)
  float f_max, tau_max;
  float inv_mass, inv_inertia[3];
  float kf_drag[3];   // 1/2 rho A_i, A = (b_y b_z, b_x b_z, b_x b_y) of the inertia box
  float kt_drag[3];   // rho / 64 b_i (b_j^4 + b_k^4)
  float c_visc_f;     // 3 pi mu d, d = mean box side
  float c_visc_t;     // pi mu d^3
  float g_eff0, dr_grav, goal_att_range;
  float w_axes[3], w_vel, w_mavg;
};

// Device status block (mirrors auv_status; first_nan_env holds INT32_MAX
// when no env has failed).
struct Status {
  int code;
  int nan_flag;
  int first_nan_env;
  int timeouts;
};

// ---------------------------------------------------------------------------
// Philox4x32-10 (Salmon et al., SC'11).  Key = (env id, seed).  Counter word
// 2 selects the stream (0 = action noise indexed by the global step,
// 1 = resets indexed by the episode), word 3 the 4-word block.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint4 philox10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                          uint32_t k0, uint32_t k1) {
#pragma unroll 1   // a rolled loop keeps the engine's hot code smaller
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = hi1 ^ c1 ^ k0, n2 = hi0 ^ c3 ^ k1;
    c0 = n0; c1 = lo1; c2 = n2; c3 = lo0;
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return make_uint4(c0, c1, c2, c3);
}

// Top 23 bits of a word, centred in their cell: exact float in (0, 1).
__device__ __forceinline__ float uniform01(uint32_t x) {
  return __fmul_rn(__uint2float_rn(((x >> 9) << 1) | 1u), 5.9604644775390625e-8f);
}

// Eight standard normals for (env, global step): two Philox blocks, Box-Muller
// on the pairs (u0,u1), (u2,u3), ...: r = sqrt(-2 ln u_even), angle 2 pi u_odd.
__device__ __forceinline__ void action_noise(uint32_t env, uint32_t seed, uint64_t t_g,
                                             float eps[8]) {
  const uint32_t lo = (uint32_t)t_g, hi = (uint32_t)(t_g >> 32);
  const uint4 a = philox10(lo, hi, 0u, 0u, env, seed);
  const uint4 b = philox10(lo, hi, 0u, 1u, env, seed);
  const uint32_t w[8] = {a.x, a.y, a.z, a.w, b.x, b.y, b.z, b.w};
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const float r = sqrtf(-2.0f * logf(uniform01(w[2 * k])));
    float s, c;
    sincospif(2.0f * uniform01(w[2 * k + 1]), &s, &c);
    eps[2 * k] = r * c;
    eps[2 * k + 1] = r * s;
  }
}

// ---------------------------------------------------------------------------
// Episode reset.  Every operation is an explicitly rounded intrinsic so that
// no contraction or reassociation changes a bit: the same steps written in
// any IEEE arithmetic give the same state.
// ---------------------------------------------------------------------------
// Maclaurin series of sine to x^15 and cosine to x^16 (|x| <= pi/2), Horner
// in x^2 with fused multiply-adds.
__device__ __forceinline__ float reset_sin(float x) {
  const float x2 = __fmul_rn(x, x);
  float p = (float)(-1.0 / 1307674368000.0);
  p = __fmaf_rn(p, x2, (float)(1.0 / 6227020800.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 39916800.0));
  p = __fmaf_rn(p, x2, (float)(1.0 / 362880.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 5040.0));
  p = __fmaf_rn(p, x2, (float)(1.0 / 120.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 6.0));
  p = __fmaf_rn(p, x2, 1.0f);
  return __fmul_rn(x, p);
}

__device__ __forceinline__ float reset_cos(float x) {
  const float x2 = __fmul_rn(x, x);
  float p = (float)(1.0 / 20922789888000.0);
  p = __fmaf_rn(p, x2, (float)(-1.0 / 87178291200.0));
  p = __fmaf_rn(p, x2, (float)(1.0 / 479001600.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 3628800.0));
  p = __fmaf_rn(p, x2, (float)(1.0 / 40320.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 720.0));
  p = __fmaf_rn(p, x2, (float)(1.0 / 24.0));
  p = __fmaf_rn(p, x2, (float)(-1.0 / 2.0));
  p = __fmaf_rn(p, x2, 1.0f);
  return p;
}

__device__ __forceinline__ float sym_draw(float u, float r) {
  return __fmaf_rn(u, __fadd_rn(r, r), -r);
}

struct Env {
  float p[3], q[4], nu[6], nup[6];
  float pd[3], qd[4], sm, sa, sd, dB, rb[3], Vc[3];
  float inv_m[6];   // 1 / diag(M_RB + M_A) for the current episode's scales
  int t_ep;
  uint32_t ep;
};

__device__ __forceinline__ void refresh_mass(const Model& M, Env& e) {
  e.inv_m[0] = 1.0f / (e.sm * M.mass + e.sa * M.added[0]);
  e.inv_m[1] = 1.0f / (e.sm * M.mass + e.sa * M.added[1]);
  e.inv_m[2] = 1.0f / (e.sm * M.mass + e.sa * M.added[2]);
  e.inv_m[3] = 1.0f / (e.sm * M.inertia[0] + e.sa * M.added[3]);
  e.inv_m[4] = 1.0f / (e.sm * M.inertia[1] + e.sa * M.added[4]);
  e.inv_m[5] = 1.0f / (e.sm * M.inertia[2] + e.sa * M.added[5]);
}

// Z-Y-X Euler composition q_z(yaw) q_y(pitch) q_x(roll) from half angles,
// every operation explicitly rounded (bit-exact reset draws).
__device__ __forceinline__ void euler_quat(float roll, float pitch, float yaw, float q[4]) {
  const float cr = reset_cos(__fmul_rn(0.5f, roll)), sr = reset_sin(__fmul_rn(0.5f, roll));
  const float cp = reset_cos(__fmul_rn(0.5f, pitch)), sp = reset_sin(__fmul_rn(0.5f, pitch));
  const float cy = reset_cos(__fmul_rn(0.5f, yaw)), sy = reset_sin(__fmul_rn(0.5f, yaw));
  const float a = __fmul_rn(cy, cp), b = __fmul_rn(sy, sp);
  const float c = __fmul_rn(cy, sp), d = __fmul_rn(sy, cp);
  q[0] = __fmaf_rn(a, cr, __fmul_rn(b, sr));
  q[1] = __fmaf_rn(a, sr, -__fmul_rn(b, cr));
  q[2] = __fmaf_rn(c, cr, __fmul_rn(d, sr));
  q[3] = __fmaf_rn(d, cr, -__fmul_rn(c, sr));
}

// New episode for env `id` at its current episode index; then episode += 1.
// Draw order: p0 xyz, roll, pitch, yaw, goal xyz, goal yaw, current xyz,
// s_m, s_a, s_d, dB, r_b xyz.
__device__ __forceinline__ void reset_env(const Model& M, uint32_t id, Env& e) {
  uint32_t w[20];
#pragma unroll
  for (int b = 0; b < 5; ++b) {
    const uint4 r = philox10(e.ep, 0u, 1u, (uint32_t)b, id, M.seed);
    w[4 * b + 0] = r.x; w[4 * b + 1] = r.y; w[4 * b + 2] = r.z; w[4 * b + 3] = r.w;
  }
  float u[20];
#pragma unroll
  for (int j = 0; j < 20; ++j) u[j] = uniform01(w[j]);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    e.p[k] = sym_draw(u[k], M.init_pos_range);
    e.pd[k] = sym_draw(u[6 + k], M.goal_pos_range);
    e.Vc[k] = sym_draw(u[10 + k], M.current_range);
  }
  const float roll = sym_draw(u[3], M.init_att_range);
  const float pitch = sym_draw(u[4], M.init_att_range);
  const float yaw = sym_draw(u[5], M.init_att_range);
  const float gyaw = sym_draw(u[9], M.goal_yaw_range);
  if (M.dr_enable) {
    const float span = __fsub_rn(M.dr_hi, M.dr_lo);
    e.sm = __fmaf_rn(u[13], span, M.dr_lo);
    e.sa = __fmaf_rn(u[14], span, M.dr_lo);
    e.sd = __fmaf_rn(u[15], span, M.dr_lo);
    e.dB = sym_draw(u[16], M.dr_buoy);
#pragma unroll
    for (int k = 0; k < 3; ++k) e.rb[k] = sym_draw(u[17 + k], M.dr_cob);
  } else {
    e.sm = 1.0f; e.sa = 1.0f; e.sd = 1.0f; e.dB = 0.0f;
    e.rb[0] = 0.0f; e.rb[1] = 0.0f; e.rb[2] = 0.0f;
  }
  euler_quat(roll, pitch, yaw, e.q);
  e.qd[0] = reset_cos(__fmul_rn(0.5f, gyaw));
  e.qd[1] = 0.0f;
  e.qd[2] = 0.0f;
  e.qd[3] = reset_sin(__fmul_rn(0.5f, gyaw));
#pragma unroll
  for (int k = 0; k < 6; ++k) { e.nu[k] = 0.0f; e.nup[k] = 0.0f; }
  e.t_ep = 0;
  e.ep += 1u;
  refresh_mass(M, e);
}

// ---------------------------------------------------------------------------
// SoA load / store (element (k, i) at k*n + i: coalesced over i).
// ---------------------------------------------------------------------------
__device__ __forceinline__ void load_env(const Model& M, const float* __restrict__ st,
                                         const float* __restrict__ pr,
                                         const int* __restrict__ t_ep,
                                         const uint32_t* __restrict__ ep, int i, Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) e.p[k] = st[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.q[k] = st[(3 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nu[k] = st[(7 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nup[k] = st[(13 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.pd[k] = pr[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.qd[k] = pr[(3 + k) * n + i];
  e.sm = pr[7 * n + i]; e.sa = pr[8 * n + i]; e.sd = pr[9 * n + i]; e.dB = pr[10 * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.rb[k] = pr[(11 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.Vc[k] = pr[(14 + k) * n + i];
  e.t_ep = t_ep[i];
  e.ep = ep[i];
  refresh_mass(M, e);
}

__device__ __forceinline__ void store_state(const Model& M, float* __restrict__ st, int i,
                                            const Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) st[k * n + i] = e.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) st[(3 + k) * n + i] = e.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) st[(7 + k) * n + i] = e.nu[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) st[(13 + k) * n + i] = e.nup[k];
}

__device__ __forceinline__ void store_env(const Model& M, float* __restrict__ st,
                                          float* __restrict__ pr, int* __restrict__ t_ep,
                                          uint32_t* __restrict__ ep, int i, const Env& e) {
  const int n = M.n;
  store_state(M, st, i, e);
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[k * n + i] = e.pd[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) pr[(3 + k) * n + i] = e.qd[k];
  pr[7 * n + i] = e.sm; pr[8 * n + i] = e.sa; pr[9 * n + i] = e.sd; pr[10 * n + i] = e.dB;
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[(11 + k) * n + i] = e.rb[k];
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[(14 + k) * n + i] = e.Vc[k];
  t_ep[i] = e.t_ep;
  ep[i] = e.ep;
}

// The per-episode parameters alone (goal, scales, buoyancy offset, centre
// of buoyancy, current), for kernels that keep them in global memory while
// the rest of the env state stays in registers.  The reload goes through L2
// (ld.global.cg): it is coherent with this thread's own earlier stores of
// the same kernel.  inv_m is not part of the arrays and is left as it is.
__device__ __forceinline__ void store_params(const Model& M, float* pr, int i, const Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[k * n + i] = e.pd[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) pr[(3 + k) * n + i] = e.qd[k];
  pr[7 * n + i] = e.sm; pr[8 * n + i] = e.sa; pr[9 * n + i] = e.sd; pr[10 * n + i] = e.dB;
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[(11 + k) * n + i] = e.rb[k];
#pragma unroll
  for (int k = 0; k < 3; ++k) pr[(14 + k) * n + i] = e.Vc[k];
}

__device__ __forceinline__ void reload_params(const Model& M, const float* pr, int i, Env& e) {
  const int n = M.n;
#pragma unroll
  for (int k = 0; k < 3; ++k) e.pd[k] = __ldcg(pr + k * n + i);
#pragma unroll
  for (int k = 0; k < 4; ++k) e.qd[k] = __ldcg(pr + (3 + k) * n + i);
  e.sm = __ldcg(pr + 7 * n + i); e.sa = __ldcg(pr + 8 * n + i);
  e.sd = __ldcg(pr + 9 * n + i); e.dB = __ldcg(pr + 10 * n + i);
#pragma unroll
  for (int k = 0; k < 3; ++k) e.rb[k] = __ldcg(pr + (11 + k) * n + i);
#pragma unroll
  for (int k = 0; k < 3; ++k) e.Vc[k] = __ldcg(pr + (14 + k) * n + i);
}

// ---------------------------------------------------------------------------
// Dynamics
// ---------------------------------------------------------------------------
// Rotation matrix (body -> world) of a unit quaternion (w, x, y, z).
__device__ __forceinline__ void quat_rot(const float q[4], float R[3][3]) {
  const float w = q[0], x = q[1], y = q[2], z = q[3];
  const float xx = x * x, yy = y * y, zz = z * z;
  const float xy = x * y, xz = x * z, yz = y * z, wx = w * x, wy = w * y, wz = w * z;
  R[0][0] = 1.0f - 2.0f * (yy + zz); R[0][1] = 2.0f * (xy - wz); R[0][2] = 2.0f * (xz + wy);
  R[1][0] = 2.0f * (xy + wz); R[1][1] = 1.0f - 2.0f * (xx + zz); R[1][2] = 2.0f * (yz - wx);
  R[2][0] = 2.0f * (xz - wy); R[2][1] = 2.0f * (yz + wx); R[2][2] = 1.0f - 2.0f * (xx + yy);
}

__device__ __forceinline__ void cross3(const float a[3], const float b[3], float o[3]) {
  o[0] = a[1] * b[2] - a[2] * b[1];
  o[1] = a[2] * b[0] - a[0] * b[2];
  o[2] = a[0] * b[1] - a[1] * b[0];
}

// Body wrench from normalised thruster commands: alloc (thrust_max clip(a)).
// Returns the clipped commands in a_c.
__device__ __forceinline__ void allocate(const Model& M, const float a[kAct], float a_c[kAct],
                                         float tau[6]) {
#pragma unroll
  for (int k = 0; k < kAct; ++k) a_c[k] = fminf(fmaxf(a[k], -1.0f), 1.0f);
#pragma unroll
  for (int r = 0; r < 6; ++r) {
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < kAct; ++k) s = fmaf(M.alloc_t[r * kAct + k], a_c[k], s);
    tau[r] = s;
  }
}

// Pose part of a semi-implicit Euler substep, shared by both models:
// p += h R v (R: attitude at the start of the substep, v: new velocity), then
// q = normalize(q (x) (cos a, sin(a) w/|w|)), a = h |w| / 2.
__device__ __forceinline__ void advance_pose(float h, const float R[3][3], const float nu[6],
                                             float p[3], float q[4]) {
#pragma unroll
  for (int i = 0; i < 3; ++i)
    p[i] = fmaf(h, R[i][0] * nu[0] + R[i][1] * nu[1] + R[i][2] * nu[2], p[i]);
  const float hw0 = 0.5f * h * nu[3], hw1 = 0.5f * h * nu[4], hw2 = 0.5f * h * nu[5];
  const float a2 = hw0 * hw0 + hw1 * hw1 + hw2 * hw2;
  float ca, sa_over_a;
  if (a2 < 0.0625f) {
    // cos a = 1 - a^2/2 + a^4/24 - a^6/720 + a^8/40320;
    // sin(a)/a = 1 - a^2/6 + a^4/120 - a^6/5040 + a^8/362880 (|a| < 1/4)
    ca = fmaf(fmaf(fmaf(fmaf(a2, 1.0f / 40320.0f, -1.0f / 720.0f), a2, 1.0f / 24.0f), a2, -0.5f),
              a2, 1.0f);
    sa_over_a = fmaf(fmaf(fmaf(fmaf(a2, 1.0f / 362880.0f, -1.0f / 5040.0f), a2, 1.0f / 120.0f),
                          a2, -1.0f / 6.0f), a2, 1.0f);
  } else {
    const float a = sqrtf(a2);
    float s;
    sincosf(a, &s, &ca);
    sa_over_a = s / a;
  }
  const float d1 = sa_over_a * hw0, d2 = sa_over_a * hw1, d3 = sa_over_a * hw2;
  const float qw = q[0], qx = q[1], qy = q[2], qz = q[3];
  float nw = qw * ca - qx * d1 - qy * d2 - qz * d3;
  float nx = qw * d1 + qx * ca + qy * d3 - qz * d2;
  float ny = qw * d2 - qx * d3 + qy * ca + qz * d1;
  float nz = qw * d3 + qx * d2 - qy * d1 + qz * ca;
  const float inv = rsqrtf(nw * nw + nx * nx + ny * ny + nz * nz);
  q[0] = nw * inv; q[1] = nx * inv; q[2] = ny * inv; q[3] = nz * inv;
}

// One semi-implicit Euler substep of
//   (M_RB + M_A) nu' = tau - C_RB(nu) nu - C_A(nu_r) nu_r - D(nu_r) nu_r
//                      + restoring + M_A nu_c'
// then p += h R v+, q = normalize(q exp(h w+ / 2)).
__device__ __forceinline__ void substep(const Model& M, Env& e, const float tau[6]) {
  float R[3][3];
  quat_rot(e.q, R);
  const float v[3] = {e.nu[0], e.nu[1], e.nu[2]};
  const float w[3] = {e.nu[3], e.nu[4], e.nu[5]};
  // current and gravity direction in the body frame: R^T V_c, R^T g_hat
  float vc[3], kb[3];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    vc[i] = R[0][i] * e.Vc[0] + R[1][i] * e.Vc[1] + R[2][i] * e.Vc[2];
    kb[i] = R[0][i] * M.ghat[0] + R[1][i] * M.ghat[1] + R[2][i] * M.ghat[2];
  }
  const float vr[3] = {v[0] - vc[0], v[1] - vc[1], v[2] - vc[2]};
  const float m = e.sm * M.mass;
  // rigid-body Coriolis [m (w x v); w x (I w)]
  float wxv[3], Iw[3], wxIw[3];
  cross3(w, v, wxv);
  Iw[0] = e.sm * M.inertia[0] * w[0];
  Iw[1] = e.sm * M.inertia[1] * w[1];
  Iw[2] = e.sm * M.inertia[2] * w[2];
  cross3(w, Iw, wxIw);
  // added-mass Coriolis [w x (A1 v_r); v_r x (A1 v_r) + w x (A2 w)]
  float A1vr[3], A2w[3], c0[3], c1[3], c2[3];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    A1vr[k] = e.sa * M.added[k] * vr[k];
    A2w[k] = e.sa * M.added[3 + k] * w[k];
  }
  cross3(w, A1vr, c0);
  cross3(vr, A1vr, c1);
  cross3(w, A2w, c2);
  // body-frame current acceleration -(w x v_c)
  float wxvc[3];
  cross3(w, vc, wxvc);
  // restoring: net force -dB k, buoyancy moment r_b x (-B k), B = m |g| + dB
  const float B = m * M.gnorm + e.dB;
  float rbxk[3];
  cross3(e.rb, kb, rbxk);
  const float nur[6] = {vr[0], vr[1], vr[2], w[0], w[1], w[2]};
  // Damping and the velocity update are the same for all six axes: two axes
  // per packed fp32 instruction (each lane rounded as the scalar operation).
  float damp[6];
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const float2 an = make_float2(fabsf(nur[2 * j]), fabsf(nur[2 * j + 1]));
    float2 t = __ffma2_rn(make_float2(M.dquad[2 * j], M.dquad[2 * j + 1]), an,
                          make_float2(M.dlin[2 * j], M.dlin[2 * j + 1]));
    t = __fmul2_rn(make_float2(e.sd, e.sd), t);
    t = __fmul2_rn(t, make_float2(nur[2 * j], nur[2 * j + 1]));
    damp[2 * j] = t.x;
    damp[2 * j + 1] = t.y;
  }
  float rhs[6];
#pragma unroll
  for (int k = 0; k < 3; ++k)
    rhs[k] = tau[k] - m * wxv[k] - c0[k] - damp[k] - e.dB * kb[k] - e.sa * M.added[k] * wxvc[k];
#pragma unroll
  for (int k = 0; k < 3; ++k)
    rhs[3 + k] = tau[3 + k] - wxIw[k] - c1[k] - c2[k] - damp[3 + k] - B * rbxk[k];
  const float2 h2 = make_float2(M.h, M.h);
#pragma unroll
  for (int j = 0; j < 3; ++j) {
    const float2 nv = __ffma2_rn(h2, __fmul2_rn(make_float2(rhs[2 * j], rhs[2 * j + 1]),
                                                make_float2(e.inv_m[2 * j], e.inv_m[2 * j + 1])),
                                 make_float2(e.nu[2 * j], e.nu[2 * j + 1]));
    e.nu[2 * j] = nv.x;
    e.nu[2 * j + 1] = nv.y;
  }
  advance_pose(M.h, R, e.nu, e.p, e.q);
}

// q_e = conj(q_d) (x) q: attitude of the body in the goal frame.
__device__ __forceinline__ void attitude_error(const Env& e, float qe[4]) {
  const float aw = e.qd[0], ax = -e.qd[1], ay = -e.qd[2], az = -e.qd[3];
  const float bw = e.q[0], bx = e.q[1], by = e.q[2], bz = e.q[3];
  qe[0] = aw * bw - ax * bx - ay * by - az * bz;
  qe[1] = aw * bx + ax * bw + ay * bz - az * by;
  qe[2] = aw * by - ax * bz + ay * bw + az * bx;
  qe[3] = aw * bz + ax * by - ay * bx + az * bw;
}

// Observation (paper §IV-B1 with the rotation-matrix error of §V-A3):
// [R(q)^T (p - p_d), R(q_e) column-major, v, w].
__device__ __forceinline__ void observe(const Env& e, float o[kObs]) {
  float R[3][3];
  quat_rot(e.q, R);
  const float dp[3] = {e.p[0] - e.pd[0], e.p[1] - e.pd[1], e.p[2] - e.pd[2]};
#pragma unroll
  for (int i = 0; i < 3; ++i) o[i] = R[0][i] * dp[0] + R[1][i] * dp[1] + R[2][i] * dp[2];
  float qe[4], Re[3][3];
  attitude_error(e, qe);
  quat_rot(qe, Re);
#pragma unroll
  for (int j = 0; j < 3; ++j)
#pragma unroll
    for (int i = 0; i < 3; ++i) o[3 + 3 * j + i] = Re[i][j];
#pragma unroll
  for (int k = 0; k < 6; ++k) o[12 + k] = e.nu[k];
}

// Reward on the post-step state: -w_pos |p - p_d| - w_att theta_e
// - w_act |a_c|^2 - w_vs |nu - nu_prev|^2, theta_e = 2 atan2(|q_e,xyz|, |q_e,w|).
__device__ __forceinline__ float reward(const Model& M, const Env& e, const float a_c[kAct]) {
  const float dx = e.p[0] - e.pd[0], dy = e.p[1] - e.pd[1], dz = e.p[2] - e.pd[2];
  const float dist = sqrtf(dx * dx + dy * dy + dz * dz);
  float qe[4];
  attitude_error(e, qe);
  const float theta = 2.0f * atan2f(sqrtf(qe[1] * qe[1] + qe[2] * qe[2] + qe[3] * qe[3]),
                                    fabsf(qe[0]));
  float a2 = 0.0f;
#pragma unroll
  for (int k = 0; k < kAct; ++k) a2 = fmaf(a_c[k], a_c[k], a2);
  float v2 = 0.0f;
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    const float d = e.nu[k] - e.nup[k];
    v2 = fmaf(d, d, v2);
  }
  return -M.w_pos * dist - M.w_att * theta - M.w_act * a2 - M.w_vs * v2;
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

__device__ __forceinline__ void flag_nan(Status* st, int env) {
  atomicExch(&st->nan_flag, 1);
  atomicMin(&st->first_nan_env, env);
  atomicCAS(&st->code, 0, -5);
}

// Physics part of one control step with action a: allocation, nu_prev,
// substeps, reward, episode bookkeeping and auto-reset.  Returns the reward;
// *done set on the episode's last step.
__device__ __forceinline__ float physics_step(const Model& M, uint32_t id, Env& e,
                                              const float a[kAct], bool* done) {
  float a_c[kAct], tau[6];
  allocate(M, a, a_c, tau);
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nup[k] = e.nu[k];
  for (int s = 0; s < M.substeps; ++s) substep(M, e, tau);
  const float r = reward(M, e, a_c);
  e.t_ep += 1;
  *done = (e.t_ep == M.episode_len);
  if (*done) reset_env(M, id, e);
  return r;
}

}  // namespace auv
