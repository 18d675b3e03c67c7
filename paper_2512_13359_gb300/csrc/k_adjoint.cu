// k_adjoint.cu -- reverse-mode adjoint of the fused control step over a
// window of actions: the back-propagation through the dynamics that SHAC
// (paper §III-A: short-horizon actor-critic, Xu et al. 2022) runs between a
// window's rewards, its terminal critic and the actions.
//
// Objective of one env over a window of T control steps taken from its
// current state x_0 = (p, q, nu) with actions a_0 .. a_{T-1}:
//   J = sum_t coef_t r_t + <lam_T, x_T>
// (r_t the step's reward, x_T the state after the last step).  The kernel
// returns dJ/da_t for every step and dJ/dx_0.  An episode end inside the
// window replaces the state by a fresh reset draw, so nothing before it
// reaches later rewards or x_T.
//
// One thread per env.  A forward pass re-simulates the window with the
// rollout's own step (auv_device.cuh) and keeps every step's input state and
// episode parameters in a scratch array [T][30][N]; the backward pass walks
// t = T-1 .. 0, re-runs step t's substeps from its stored input to recover
// the substep inputs (registers / local memory, S <= 8), and applies the
// vector-Jacobian product of each piece in reverse: reward, substeps (pose
// update, velocity update, the right-hand side of the equations of motion),
// allocation and the command clip.  The env's buffers are read, not written.
#include "auv_kernels.h"
#include "paper_device.cuh"

namespace auv {

namespace {

constexpr int kAdjThreads = 128;
constexpr int kX = 13;          // p(3) q(4) nu(6)
constexpr int kScratchF = 30;   // x(13) pd(3) qd(4) sm sa sd dB rb(3) Vc(3)

struct X {
  float p[3], q[4], nu[6];
};

__device__ __forceinline__ void save_step(float* __restrict__ sc, size_t n, int i, const Env& e) {
  float v[kScratchF] = {e.p[0], e.p[1], e.p[2], e.q[0], e.q[1], e.q[2], e.q[3],
                        e.nu[0], e.nu[1], e.nu[2], e.nu[3], e.nu[4], e.nu[5],
                        e.pd[0], e.pd[1], e.pd[2], e.qd[0], e.qd[1], e.qd[2], e.qd[3],
                        e.sm, e.sa, e.sd, e.dB, e.rb[0], e.rb[1], e.rb[2],
                        e.Vc[0], e.Vc[1], e.Vc[2]};
#pragma unroll
  for (int k = 0; k < kScratchF; ++k) sc[k * n + i] = v[k];
}

__device__ __forceinline__ void load_step(const Model& M, const float* __restrict__ sc, size_t n,
                                          int i, Env& e) {
  float v[kScratchF];
#pragma unroll
  for (int k = 0; k < kScratchF; ++k) v[k] = sc[k * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.p[k] = v[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.q[k] = v[3 + k];
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nu[k] = v[7 + k];
#pragma unroll
  for (int k = 0; k < 3; ++k) e.pd[k] = v[13 + k];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.qd[k] = v[16 + k];
  e.sm = v[20]; e.sa = v[21]; e.sd = v[22]; e.dB = v[23];
#pragma unroll
  for (int k = 0; k < 3; ++k) { e.rb[k] = v[24 + k]; e.Vc[k] = v[27 + k]; }
  refresh_mass(M, e);
}

__device__ __forceinline__ void get_x(const Env& e, X& x) {
#pragma unroll
  for (int k = 0; k < 3; ++k) x.p[k] = e.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) x.q[k] = e.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) x.nu[k] = e.nu[k];
}

__device__ __forceinline__ void put_x(const X& x, Env& e) {
#pragma unroll
  for (int k = 0; k < 3; ++k) e.p[k] = x.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) e.q[k] = x.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) e.nu[k] = x.nu[k];
}

// lam_a += b x lam_y and lam_b += lam_y x a, for y = a x b.
__device__ __forceinline__ void cross_vjp(const float a[3], const float b[3], const float ly[3],
                                          float la[3], float lb[3]) {
  float t[3];
  cross3(b, ly, t);
#pragma unroll
  for (int k = 0; k < 3; ++k) la[k] += t[k];
  cross3(ly, a, t);
#pragma unroll
  for (int k = 0; k < 3; ++k) lb[k] += t[k];
}

// lam_q += (dR(q)/dq)^T : lam_R for the rotation matrix of quat_rot.
__device__ __forceinline__ void rot_vjp(const float q[4], const float L[3][3], float lq[4]) {
  const float w = q[0], x = q[1], y = q[2], z = q[3];
  lq[0] += 2.0f * (-z * L[0][1] + y * L[0][2] + z * L[1][0] - x * L[1][2] - y * L[2][0] +
                   x * L[2][1]);
  lq[1] += 2.0f * (y * L[0][1] + z * L[0][2] + y * L[1][0] - 2.0f * x * L[1][1] - w * L[1][2] +
                   z * L[2][0] + w * L[2][1] - 2.0f * x * L[2][2]);
  lq[2] += 2.0f * (-2.0f * y * L[0][0] + x * L[0][1] + w * L[0][2] + x * L[1][0] + z * L[1][2] -
                   w * L[2][0] + z * L[2][1] - 2.0f * y * L[2][2]);
  lq[3] += 2.0f * (-2.0f * z * L[0][0] - w * L[0][1] + x * L[0][2] + w * L[1][0] -
                   2.0f * z * L[1][1] + y * L[1][2] + x * L[2][0] + y * L[2][1]);
}

// Vector-Jacobian product of the pose part of a substep (auv_device.cuh:
// advance_pose, shared by both models): p1 = p + h R(q) v1 and
// q1 = normalize(q (x) (cos a, sin(a)/a hw)), hw = h w1 / 2, a = |hw|.  On
// entry lx holds dJ/d(p1, q1, nu1); on exit lnu1 = dJ/dnu1 (the direct part
// plus the pose's), LR = dJ/dR from the position update, lq = dJ/dq from the
// attitude product; lx.p is unchanged (p1 = p + ...).
__device__ void pose_vjp(float h, const float q[4], const float R[3][3], const float nu1[6],
                         const X& lx, float lnu1[6], float LR[3][3], float lq[4]) {
  const float hw[3] = {0.5f * h * nu1[3], 0.5f * h * nu1[4], 0.5f * h * nu1[5]};
  const float a2 = hw[0] * hw[0] + hw[1] * hw[1] + hw[2] * hw[2];
  float ca, s, g;     // cos a, sin(a)/a, (a cos a - sin a)/a^3
  if (a2 < 0.25f) {
    ca = fmaf(fmaf(fmaf(fmaf(a2, 1.0f / 40320.0f, -1.0f / 720.0f), a2, 1.0f / 24.0f), a2, -0.5f),
              a2, 1.0f);
    s = fmaf(fmaf(fmaf(fmaf(a2, 1.0f / 362880.0f, -1.0f / 5040.0f), a2, 1.0f / 120.0f), a2,
                  -1.0f / 6.0f),
             a2, 1.0f);
    g = fmaf(fmaf(fmaf(fmaf(a2, -1.0f / 3991680.0f, 1.0f / 45360.0f), a2, -1.0f / 840.0f), a2,
                  1.0f / 30.0f),
             a2, -1.0f / 3.0f);
  } else {
    const float a = sqrtf(a2);
    float sn;
    sincosf(a, &sn, &ca);
    s = sn / a;
    g = (a * ca - sn) / (a2 * a);
  }
  const float d[4] = {ca, s * hw[0], s * hw[1], s * hw[2]};
  const float qw = q[0], qx = q[1], qy = q[2], qz = q[3];
  const float u[4] = {qw * d[0] - qx * d[1] - qy * d[2] - qz * d[3],
                      qw * d[1] + qx * d[0] + qy * d[3] - qz * d[2],
                      qw * d[2] - qx * d[3] + qy * d[0] + qz * d[1],
                      qw * d[3] + qx * d[2] - qy * d[1] + qz * d[0]};
  const float inv_u = rsqrtf(u[0] * u[0] + u[1] * u[1] + u[2] * u[2] + u[3] * u[3]);
  const float q1[4] = {u[0] * inv_u, u[1] * inv_u, u[2] * inv_u, u[3] * inv_u};
  // q1 = u / |u|
  const float dot = lx.q[0] * q1[0] + lx.q[1] * q1[1] + lx.q[2] * q1[2] + lx.q[3] * q1[3];
  float lu[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) lu[k] = (lx.q[k] - dot * q1[k]) * inv_u;
  // u = q (x) d
  lq[0] = d[0] * lu[0] + d[1] * lu[1] + d[2] * lu[2] + d[3] * lu[3];
  lq[1] = -d[1] * lu[0] + d[0] * lu[1] - d[3] * lu[2] + d[2] * lu[3];
  lq[2] = -d[2] * lu[0] + d[3] * lu[1] + d[0] * lu[2] - d[1] * lu[3];
  lq[3] = -d[3] * lu[0] - d[2] * lu[1] + d[1] * lu[2] + d[0] * lu[3];
  const float ld0 = qw * lu[0] + qx * lu[1] + qy * lu[2] + qz * lu[3];
  const float ld[3] = {-qx * lu[0] + qw * lu[1] + qz * lu[2] - qy * lu[3],
                       -qy * lu[0] - qz * lu[1] + qw * lu[2] + qx * lu[3],
                       -qz * lu[0] + qy * lu[1] - qx * lu[2] + qw * lu[3]};
  // d = (cos a, s(a) hw), a = |hw|
  const float hl = hw[0] * ld[0] + hw[1] * ld[1] + hw[2] * ld[2];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    const float lhw = -s * hw[k] * ld0 + s * ld[k] + g * hw[k] * hl;
    lnu1[3 + k] = lx.nu[3 + k] + 0.5f * h * lhw;
  }
  // p1 = p + h R v1
#pragma unroll
  for (int i = 0; i < 3; ++i) {
#pragma unroll
    for (int j = 0; j < 3; ++j) LR[i][j] = h * lx.p[i] * nu1[j];
  }
#pragma unroll
  for (int j = 0; j < 3; ++j)
    lnu1[j] = lx.nu[j] + h * (R[0][j] * lx.p[0] + R[1][j] * lx.p[1] + R[2][j] * lx.p[2]);
}

// Vector-Jacobian product of one substep (auv_device.cuh: substep) taken
// from input x with wrench tau: on entry lx is dJ/d(output), on exit
// dJ/d(input); ltau accumulates dJ/dtau.
__device__ void substep_vjp(const Model& M, const Env& e, const X& x, const float tau[6],
                            X& lx, float ltau[6]) {
  // ---- recompute the forward quantities of the substep ----
  float R[3][3];
  quat_rot(x.q, R);
  const float v[3] = {x.nu[0], x.nu[1], x.nu[2]};
  const float w[3] = {x.nu[3], x.nu[4], x.nu[5]};
  float vc[3], kb[3];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    vc[i] = R[0][i] * e.Vc[0] + R[1][i] * e.Vc[1] + R[2][i] * e.Vc[2];
    kb[i] = R[0][i] * M.ghat[0] + R[1][i] * M.ghat[1] + R[2][i] * M.ghat[2];
  }
  const float vr[3] = {v[0] - vc[0], v[1] - vc[1], v[2] - vc[2]};
  const float m = e.sm * M.mass;
  const float I[3] = {e.sm * M.inertia[0], e.sm * M.inertia[1], e.sm * M.inertia[2]};
  const float A1[3] = {e.sa * M.added[0], e.sa * M.added[1], e.sa * M.added[2]};
  const float A2[3] = {e.sa * M.added[3], e.sa * M.added[4], e.sa * M.added[5]};
  float wxv[3], Iw[3], wxIw[3], A1vr[3], A2w[3], c0[3], c1[3], c2[3], wxvc[3], rbxk[3];
  cross3(w, v, wxv);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    Iw[k] = I[k] * w[k];
    A1vr[k] = A1[k] * vr[k];
    A2w[k] = A2[k] * w[k];
  }
  cross3(w, Iw, wxIw);
  cross3(w, A1vr, c0);
  cross3(vr, A1vr, c1);
  cross3(w, A2w, c2);
  cross3(w, vc, wxvc);
  const float B = m * M.gnorm + e.dB;
  cross3(e.rb, kb, rbxk);
  const float nur[6] = {vr[0], vr[1], vr[2], w[0], w[1], w[2]};
  float rhs[6], nu1[6];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    const float dl = e.sd * (M.dlin[k] + M.dquad[k] * fabsf(nur[k])) * nur[k];
    rhs[k] = tau[k] - m * wxv[k] - c0[k] - dl - e.dB * kb[k] - A1[k] * wxvc[k];
    const float da = e.sd * (M.dlin[3 + k] + M.dquad[3 + k] * fabsf(nur[3 + k])) * nur[3 + k];
    rhs[3 + k] = tau[3 + k] - wxIw[k] - c1[k] - c2[k] - da - B * rbxk[k];
  }
#pragma unroll
  for (int k = 0; k < 6; ++k) nu1[k] = x.nu[k] + M.h * (rhs[k] * e.inv_m[k]);
  float lnu1[6], LR[3][3], lq[4];
  pose_vjp(M.h, x.q, R, nu1, lx, lnu1, LR, lq);
  // nu1 = nu + h M^-1 rhs
  float lr[6];
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    lr[k] = M.h * e.inv_m[k] * lnu1[k];
    ltau[k] += lr[k];
  }
  const float Ll[3] = {lr[0], lr[1], lr[2]}, La[3] = {lr[3], lr[4], lr[5]};
  float lv[3] = {0.f, 0.f, 0.f}, lw[3] = {0.f, 0.f, 0.f}, lvr[3] = {0.f, 0.f, 0.f};
  float lvc[3] = {0.f, 0.f, 0.f}, lkb[3] = {0.f, 0.f, 0.f};
  float ly[3], lt[3];
  // -m (w x v)
#pragma unroll
  for (int k = 0; k < 3; ++k) ly[k] = -m * Ll[k];
  cross_vjp(w, v, ly, lw, lv);
  // -(w x A1 vr)
#pragma unroll
  for (int k = 0; k < 3; ++k) { ly[k] = -Ll[k]; lt[k] = 0.f; }
  cross_vjp(w, A1vr, ly, lw, lt);
#pragma unroll
  for (int k = 0; k < 3; ++k) lvr[k] += A1[k] * lt[k];
  // -dB kb and -A1 (w x vc)
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lkb[k] -= e.dB * Ll[k];
    ly[k] = -A1[k] * Ll[k];
  }
  cross_vjp(w, vc, ly, lw, lvc);
  // -(w x I w)
#pragma unroll
  for (int k = 0; k < 3; ++k) { ly[k] = -La[k]; lt[k] = 0.f; }
  cross_vjp(w, Iw, ly, lw, lt);
#pragma unroll
  for (int k = 0; k < 3; ++k) lw[k] += I[k] * lt[k];
  // -(vr x A1 vr)
#pragma unroll
  for (int k = 0; k < 3; ++k) lt[k] = 0.f;
  cross_vjp(vr, A1vr, ly, lvr, lt);
#pragma unroll
  for (int k = 0; k < 3; ++k) lvr[k] += A1[k] * lt[k];
  // -(w x A2 w)
#pragma unroll
  for (int k = 0; k < 3; ++k) lt[k] = 0.f;
  cross_vjp(w, A2w, ly, lw, lt);
#pragma unroll
  for (int k = 0; k < 3; ++k) lw[k] += A2[k] * lt[k];
  // -B (rb x kb): only kb depends on the state
  {
    float t[3];
    cross3(La, e.rb, t);
#pragma unroll
    for (int k = 0; k < 3; ++k) lkb[k] -= B * t[k];
  }
  // damping on the relative velocity
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lvr[k] -= Ll[k] * e.sd * (M.dlin[k] + 2.0f * M.dquad[k] * fabsf(nur[k]));
    lw[k] -= La[k] * e.sd * (M.dlin[3 + k] + 2.0f * M.dquad[3 + k] * fabsf(nur[3 + k]));
  }
  // vr = v - vc;  vc = R^T V_c,  kb = R^T g_hat
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lv[k] += lvr[k];
    lvc[k] -= lvr[k];
  }
#pragma unroll
  for (int j = 0; j < 3; ++j) {
#pragma unroll
    for (int i = 0; i < 3; ++i) LR[j][i] += lvc[i] * e.Vc[j] + lkb[i] * M.ghat[j];
  }
  rot_vjp(x.q, LR, lq);
  // outputs: dJ/d(input)
#pragma unroll
  for (int k = 0; k < 4; ++k) lx.q[k] = lq[k];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lx.nu[k] = lnu1[k] + lv[k];
    lx.nu[3 + k] = lnu1[3 + k] + lw[k];
  }
  // lx.p passes through (p1 = p + ...)
}

// Adds coef * dr/d(post-step state) to lx and returns dr/dnu_prev (scaled)
// in lnup and coef * dr/da_c in la.
__device__ void reward_vjp(const Model& M, const Env& e, const float a_c[kAct],
                           const float nup[6], float coef, X& lx, float lnup[6],
                           float la[kAct]) {
  const float dx[3] = {e.p[0] - e.pd[0], e.p[1] - e.pd[1], e.p[2] - e.pd[2]};
  const float dist = sqrtf(dx[0] * dx[0] + dx[1] * dx[1] + dx[2] * dx[2]);
  if (dist > 0.0f) {
    const float c = -coef * M.w_pos / dist;
#pragma unroll
    for (int k = 0; k < 3; ++k) lx.p[k] += c * dx[k];
  }
  float qe[4];
  attitude_error(e, qe);
  const float vn = sqrtf(qe[1] * qe[1] + qe[2] * qe[2] + qe[3] * qe[3]);
  const float s0 = fabsf(qe[0]);
  const float den = vn * vn + s0 * s0;
  float lqe[4] = {0.f, 0.f, 0.f, 0.f};
  if (den > 0.0f) {
    const float c = -coef * M.w_att * 2.0f / den;
    lqe[0] = c * (-vn) * (qe[0] < 0.0f ? -1.0f : 1.0f);
    if (vn > 0.0f) {
      const float cv = c * s0 / vn;
      lqe[1] = cv * qe[1];
      lqe[2] = cv * qe[2];
      lqe[3] = cv * qe[3];
    }
  }
  // qe = conj(q_d) (x) q
  const float aw = e.qd[0], ax = -e.qd[1], ay = -e.qd[2], az = -e.qd[3];
  lx.q[0] += aw * lqe[0] + ax * lqe[1] + ay * lqe[2] + az * lqe[3];
  lx.q[1] += -ax * lqe[0] + aw * lqe[1] + az * lqe[2] - ay * lqe[3];
  lx.q[2] += -ay * lqe[0] - az * lqe[1] + aw * lqe[2] + ax * lqe[3];
  lx.q[3] += -az * lqe[0] + ay * lqe[1] - ax * lqe[2] + aw * lqe[3];
#pragma unroll
  for (int k = 0; k < kAct; ++k) la[k] = -coef * M.w_act * 2.0f * a_c[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    const float dv = -coef * M.w_vs * 2.0f * (e.nu[k] - nup[k]);
    lx.nu[k] += dv;
    lnup[k] = -dv;
  }
}

__global__ void __launch_bounds__(kAdjThreads, 4) k_adjoint(
    const Model M, Buffers B, const float* __restrict__ act, int T,
    const float* __restrict__ coef, const float* __restrict__ lam_T, float* __restrict__ g_act,
    float* __restrict__ lam_0, float* __restrict__ rew, uint8_t* __restrict__ done,
    float* __restrict__ scratch, Status* st) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  const uint32_t id = M.id_base + (uint32_t)i;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  uint64_t ends = 0;
  // Step t + 1's actions are loaded while step t integrates (and step t - 1's
  // while the reverse sweep differentiates step t).
  float a_next[kAct];
#pragma unroll
  for (int k = 0; k < kAct; ++k) a_next[k] = T > 0 ? __ldg(act + (size_t)k * n + i) : 0.0f;
  for (int t = 0; t < T; ++t) {
    save_step(scratch + (size_t)t * kScratchF * n, n, i, e);
    float a[kAct];
#pragma unroll
    for (int k = 0; k < kAct; ++k) a[k] = a_next[k];
    if (t + 1 < T) {
#pragma unroll
      for (int k = 0; k < kAct; ++k)
        a_next[k] = __ldg(act + ((size_t)(t + 1) * kAct + k) * n + i);
    }
    bool d;
    const float r = physics_step(M, id, e, a, &d);
    if (d) ends |= 1ull << t;
    if (rew) rew[(size_t)t * n + i] = r;
    if (done) done[(size_t)t * n + i] = d ? 1 : 0;
  }
  X lx;
#pragma unroll
  for (int k = 0; k < kX; ++k) {
    const float v = lam_T ? __ldg(lam_T + k * n + i) : 0.0f;
    if (k < 3) lx.p[k] = v;
    else if (k < 7) lx.q[k - 3] = v;
    else lx.nu[k - 7] = v;
  }
  X xs[8];
#pragma unroll
  for (int k = 0; k < kAct; ++k)
    a_next[k] = T > 0 ? __ldg(act + ((size_t)(T - 1) * kAct + k) * n + i) : 0.0f;
  for (int t = T - 1; t >= 0; --t) {
    if ((ends >> t) & 1ull) {
#pragma unroll
      for (int k = 0; k < 3; ++k) lx.p[k] = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k) lx.q[k] = 0.f;
#pragma unroll
      for (int k = 0; k < 6; ++k) lx.nu[k] = 0.f;
    }
    Env es;
    load_step(M, scratch + (size_t)t * kScratchF * n, n, i, es);
    float a[kAct], a_c[kAct], tau[6], nup[6];
#pragma unroll
    for (int k = 0; k < kAct; ++k) a[k] = a_next[k];
    if (t > 0) {
#pragma unroll
      for (int k = 0; k < kAct; ++k) a_next[k] = __ldg(act + ((size_t)(t - 1) * kAct + k) * n + i);
    }
    allocate(M, a, a_c, tau);
#pragma unroll
    for (int k = 0; k < 6; ++k) nup[k] = es.nu[k];
    for (int s = 0; s < M.substeps; ++s) {
      get_x(es, xs[s]);
      substep(M, es, tau);
    }
    float la[kAct], lnup[6], ltau[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    reward_vjp(M, es, a_c, nup, __ldg(coef + t), lx, lnup, la);
    for (int s = M.substeps - 1; s >= 0; --s) {
      put_x(xs[s], es);
      substep_vjp(M, es, xs[s], tau, lx, ltau);
    }
#pragma unroll
    for (int k = 0; k < 6; ++k) lx.nu[k] += lnup[k];
#pragma unroll
    for (int k = 0; k < kAct; ++k) {
      float g = la[k];
#pragma unroll
      for (int r = 0; r < 6; ++r) g = fmaf(M.alloc_t[r * kAct + k], ltau[r], g);
      // the clip passes a through on [-1, 1] (the subgradient 1 at the edges)
      g_act[((size_t)t * kAct + k) * n + i] = (a[k] >= -1.0f && a[k] <= 1.0f) ? g : 0.0f;
    }
  }
  float out[kX] = {lx.p[0], lx.p[1], lx.p[2], lx.q[0], lx.q[1], lx.q[2], lx.q[3],
                   lx.nu[0], lx.nu[1], lx.nu[2], lx.nu[3], lx.nu[4], lx.nu[5]};
  float s = 0.0f;
#pragma unroll
  for (int k = 0; k < kX; ++k) s += out[k];
  if (!isfinite(s)) flag_nan(st, i);
  if (lam_0) {
#pragma unroll
    for (int k = 0; k < kX; ++k) lam_0[k * n + i] = out[k];
  }
}

// ---------------------------------------------------------------------------
// SHAC in closed loop: the window's steps one at a time, with the policy
// network's products done outside (k_gemm.cu) between these kernels.
// ---------------------------------------------------------------------------

// dJ/d(state) += (d obs / d state)^T lo for the observation of auv_device.cuh.
__device__ void obs_vjp(const Env& e, const float lo[kObs], X& lx) {
  float R[3][3];
  quat_rot(e.q, R);
  const float dp[3] = {e.p[0] - e.pd[0], e.p[1] - e.pd[1], e.p[2] - e.pd[2]};
  float LR[3][3];
#pragma unroll
  for (int j = 0; j < 3; ++j) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
      LR[j][i] = lo[i] * dp[j];                  // o_i = sum_j R[j][i] dp_j
      lx.p[j] += R[j][i] * lo[i];
    }
  }
  rot_vjp(e.q, LR, lx.q);
  float qe[4], LRe[3][3];
  attitude_error(e, qe);
#pragma unroll
  for (int j = 0; j < 3; ++j) {
#pragma unroll
    for (int i = 0; i < 3; ++i) LRe[i][j] = lo[3 + 3 * j + i];   // o_{3+3j+i} = R(qe)[i][j]
  }
  float lqe[4] = {0.f, 0.f, 0.f, 0.f};
  rot_vjp(qe, LRe, lqe);
  const float aw = e.qd[0], ax = -e.qd[1], ay = -e.qd[2], az = -e.qd[3];
  lx.q[0] += aw * lqe[0] + ax * lqe[1] + ay * lqe[2] + az * lqe[3];
  lx.q[1] += -ax * lqe[0] + aw * lqe[1] + az * lqe[2] - ay * lqe[3];
  lx.q[2] += -ay * lqe[0] - az * lqe[1] + aw * lqe[2] + ax * lqe[3];
  lx.q[3] += -az * lqe[0] + ay * lqe[1] - ax * lqe[2] + aw * lqe[3];
#pragma unroll
  for (int k = 0; k < 6; ++k) lx.nu[k] += lo[12 + k];
}

__device__ __forceinline__ void load_lam(const float* __restrict__ lam, size_t n, int i, X& lx) {
#pragma unroll
  for (int k = 0; k < 3; ++k) lx.p[k] = lam[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) lx.q[k] = lam[(3 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 6; ++k) lx.nu[k] = lam[(7 + k) * n + i];
}

__device__ __forceinline__ void store_lam(float* __restrict__ lam, size_t n, int i, const X& lx) {
#pragma unroll
  for (int k = 0; k < 3; ++k) lam[k * n + i] = lx.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) lam[(3 + k) * n + i] = lx.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) lam[(7 + k) * n + i] = lx.nu[k];
}

// Reparameterised action a = mu + exp(clamp(ls)) eps from a policy head row.
__device__ __forceinline__ void shac_action(const Model& M, const float* __restrict__ y,
                                            const float eps[kAct], float a[kAct],
                                            float sig[kAct], bool in[kAct]) {
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    const float raw = y[kAct + k];
    in[k] = raw >= M.logstd_min && raw <= M.logstd_max;
    sig[k] = expf(fminf(fmaxf(raw, M.logstd_min), M.logstd_max));
    a[k] = fmaf(sig[k], eps[k], y[k]);
  }
}

// Observation row of the network input (augmented: 1 at column kObs, zeros
// up to ldx) of each env's current state; with sc, also the step's scratch.
__global__ void __launch_bounds__(kAdjThreads) k_shac_obs(const Model M, Buffers B,
                                                          float* __restrict__ sc,
                                                          float* __restrict__ X, int ldx,
                                                          float* __restrict__ obs_fm, int t) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  if (sc) save_step(sc, (size_t)M.n, i, e);
  float o[kObs];
  observe(e, o);
  float* x = X + (size_t)i * ldx;
#pragma unroll
  for (int k = 0; k < kObs; ++k) x[k] = o[k];
  x[kObs] = 1.0f;
  for (int k = kObs + 1; k < ldx; ++k) x[k] = 0.0f;
  if (obs_fm) {
#pragma unroll
    for (int k = 0; k < kObs; ++k) obs_fm[((size_t)t * kObs + k) * M.n + i] = o[k];
  }
}

// One closed-loop step from the policy head Y [N][ldy]: action, physics,
// episode bookkeeping; the env's buffers are advanced.
__global__ void __launch_bounds__(kAdjThreads) k_shac_step(const Model M, Buffers B,
                                                           const float* __restrict__ Y, int ldy,
                                                           uint64_t t_g, float* __restrict__ rew,
                                                           uint8_t* __restrict__ done,
                                                           Status* st) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  Env e;
  load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  const uint32_t id = M.id_base + (uint32_t)i;
  float eps[kAct], a[kAct], sig[kAct];
  bool in[kAct];
  action_noise(id, M.seed, t_g, eps);
  shac_action(M, Y + (size_t)i * ldy, eps, a, sig, in);
  bool d;
  const float r = physics_step(M, id, e, a, &d);
  if (!env_finite(e)) flag_nan(st, i);
  store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  rew[i] = r;
  done[i] = d ? 1 : 0;
}

// Backward of one closed-loop step: lam (dJ/d post-step state, [13][N]) is
// replaced by dJ/d pre-step state through the physics, and the policy head's
// gradient is written to gY [N][ldy] (mean, then the log-std head through
// a = mu + sigma eps; zero where the clamp is active).
__global__ void __launch_bounds__(kAdjThreads, 4) k_shac_bwd(const Model M,
                                                          const float* __restrict__ sc,
                                                          const float* __restrict__ Y, int ldy,
                                                          const uint8_t* __restrict__ done,
                                                          uint64_t t_g, const float* __restrict__ coef,
                                                          float* __restrict__ lam,
                                                          float* __restrict__ gY) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  const uint32_t id = M.id_base + (uint32_t)i;
  X lx;
  if (done[i]) {
#pragma unroll
    for (int k = 0; k < 3; ++k) lx.p[k] = 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) lx.q[k] = 0.f;
#pragma unroll
    for (int k = 0; k < 6; ++k) lx.nu[k] = 0.f;
  } else {
    load_lam(lam, n, i, lx);
  }
  Env es;
  load_step(M, sc, n, i, es);
  float eps[kAct], a[kAct], sig[kAct], a_c[kAct], tau[6], nup[6];
  bool in[kAct];
  action_noise(id, M.seed, t_g, eps);
  shac_action(M, Y + (size_t)i * ldy, eps, a, sig, in);
  allocate(M, a, a_c, tau);
#pragma unroll
  for (int k = 0; k < 6; ++k) nup[k] = es.nu[k];
  X xs[8];
  for (int s = 0; s < M.substeps; ++s) {
    get_x(es, xs[s]);
    substep(M, es, tau);
  }
  float la[kAct], lnup[6], ltau[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  reward_vjp(M, es, a_c, nup, __ldg(coef), lx, lnup, la);
  for (int s = M.substeps - 1; s >= 0; --s) substep_vjp(M, es, xs[s], tau, lx, ltau);
#pragma unroll
  for (int k = 0; k < 6; ++k) lx.nu[k] += lnup[k];
  float* g = gY + (size_t)i * ldy;
#pragma unroll
  for (int k = 0; k < kAct; ++k) {
    float ga = la[k];
#pragma unroll
    for (int r = 0; r < 6; ++r) ga = fmaf(M.alloc_t[r * kAct + k], ltau[r], ga);
    if (!(a[k] >= -1.0f && a[k] <= 1.0f)) ga = 0.0f;
    g[k] = ga;
    g[kAct + k] = in[k] ? ga * sig[k] * eps[k] : 0.0f;
  }
  store_lam(lam, n, i, lx);
}

// lam += (d obs / d state)^T gX at the state of scratch sc (or of the env's
// buffers when sc is NULL); gX [N][ldx], first kObs columns.
__global__ void __launch_bounds__(kAdjThreads) k_shac_obs_vjp(const Model M, Buffers B,
                                                              const float* __restrict__ sc,
                                                              const float* __restrict__ gX,
                                                              int ldx, float* __restrict__ lam) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  Env e;
  if (sc) {
    load_step(M, sc, n, i, e);
  } else {
    load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  }
  float lo[kObs];
#pragma unroll
  for (int k = 0; k < kObs; ++k) lo[k] = gX[(size_t)i * ldx + k];
  X lx;
  load_lam(lam, n, i, lx);
  obs_vjp(e, lo, lx);
  store_lam(lam, n, i, lx);
}

// J_i = sum_t coef_t r_t + coef_V V_i (V [N][ldv], column 0; NULL for none).
__global__ void __launch_bounds__(kAdjThreads) k_shac_objective(int n, int T,
                                                                const float* __restrict__ rew,
                                                                const float* __restrict__ coef,
                                                                const float* __restrict__ V,
                                                                int ldv, float coef_V,
                                                                float* __restrict__ J) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= n) return;
  float s = 0.0f;
  for (int t = 0; t < T; ++t) s = fmaf(__ldg(coef + t), rew[(size_t)t * n + i], s);
  if (V) s = fmaf(coef_V, V[(size_t)i * ldv], s);
  J[i] = s;
}

__global__ void __launch_bounds__(kAdjThreads) k_fill_col(int n, float* __restrict__ buf, int ld,
                                                          float v) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i < n) buf[(size_t)i * ld] = v;
}

// ---------------------------------------------------------------------------
// The paper model (paper_device.cuh): its state adds the K-slot history of
// clipped actions (rows 13 + 6 j + k), which the reward's moving-average
// term reads, so the adjoint carries those rows too.
// ---------------------------------------------------------------------------
constexpr int kPScratchF = 28;   // x(13) pd(3) qd(4) g t_ep mean of the history(6)

// lq += (d theta / dq)^T lth for the axis-angle error of paper_device.cuh:
// qe = conj(q_d) (x) q, flipped to w >= 0; theta = s v, s = 2 atan2(|v|, w) / |v|.
__device__ void att_error_vjp(const paper::Env& e, const float lth[3], float lq[4]) {
  const float aw = e.qd[0], ax = -e.qd[1], ay = -e.qd[2], az = -e.qd[3];
  const float bw = e.q[0], bx = e.q[1], by = e.q[2], bz = e.q[3];
  float w = aw * bw - ax * bx - ay * by - az * bz;
  float v[3] = {aw * bx + ax * bw + ay * bz - az * by, aw * by - ax * bz + ay * bw + az * bx,
                aw * bz + ax * by - ay * bx + az * bw};
  const float sg = w < 0.0f ? -1.0f : 1.0f;
  w *= sg;
#pragma unroll
  for (int k = 0; k < 3; ++k) v[k] *= sg;
  const float vn2 = v[0] * v[0] + v[1] * v[1] + v[2] * v[2], vn = sqrtf(vn2);
  const float den = vn2 + w * w;
  float s, c;      // s, and (ds/d|v|) / |v|
  if (vn > 1e-3f * w) {
    s = 2.0f * atan2f(vn, w) / vn;
    c = (2.0f * w / den - s) / vn2;
  } else {         // series in r = |v| / w: s = (2/w)(1 - r^2/3 + r^4/5)
    const float iw = 1.0f / w, r2 = vn2 * iw * iw;
    s = 2.0f * iw * (1.0f - r2 / 3.0f + r2 * r2 / 5.0f);
    c = 4.0f * iw * iw * iw * (-1.0f / 3.0f + 2.0f * r2 / 5.0f);
  }
  const float tv = lth[0] * v[0] + lth[1] * v[1] + lth[2] * v[2];
  float lqe[4];
  lqe[0] = sg * tv * (-2.0f / den);
#pragma unroll
  for (int k = 0; k < 3; ++k) lqe[1 + k] = sg * (s * lth[k] + tv * c * v[k]);
  lq[0] += aw * lqe[0] + ax * lqe[1] + ay * lqe[2] + az * lqe[3];
  lq[1] += -ax * lqe[0] + aw * lqe[1] + az * lqe[2] - ay * lqe[3];
  lq[2] += -ay * lqe[0] - az * lqe[1] + aw * lqe[2] + ax * lqe[3];
  lq[3] += -az * lqe[0] + ay * lqe[1] - ax * lqe[2] + aw * lqe[3];
}

// dJ/d(state) += (d obs / d state)^T lo for the paper model's observation
// [R^T (p - p_d), theta, v, w].
__device__ void paper_obs_vjp(const paper::Env& e, const float lo[paper::kObs], X& lx) {
  float R[3][3];
  quat_rot(e.q, R);
  const float dp[3] = {e.p[0] - e.pd[0], e.p[1] - e.pd[1], e.p[2] - e.pd[2]};
  float LR[3][3];
#pragma unroll
  for (int j = 0; j < 3; ++j) {
#pragma unroll
    for (int i = 0; i < 3; ++i) {
      LR[j][i] = lo[i] * dp[j];
      lx.p[j] += R[j][i] * lo[i];
    }
  }
  rot_vjp(e.q, LR, lx.q);
  att_error_vjp(e, lo + 3, lx.q);
#pragma unroll
  for (int k = 0; k < 6; ++k) lx.nu[k] += lo[6 + k];
}

// VJP of one paper-model substep (paper_device.cuh: substep).
__device__ void paper_substep_vjp(const Model& M, const paper::Env& e, const X& x,
                                  const float tau[6], X& lx, float ltau[6]) {
  float R[3][3];
  quat_rot(x.q, R);
  const float v[3] = {x.nu[0], x.nu[1], x.nu[2]};
  const float w[3] = {x.nu[3], x.nu[4], x.nu[5]};
  const float m = M.mass, mg = m * e.g;
  float wxv[3], Iw[3], wxIw[3], nu1[6];
  cross3(w, v, wxv);
#pragma unroll
  for (int k = 0; k < 3; ++k) Iw[k] = M.inertia[k] * w[k];
  cross3(w, Iw, wxIw);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    const float f = -M.kf_drag[k] * fabsf(v[k]) * v[k] - M.c_visc_f * v[k];
    const float t = -M.kt_drag[k] * fabsf(w[k]) * w[k] - M.c_visc_t * w[k];
    const float lin = tau[k] + f - mg * R[2][k] - m * wxv[k];
    const float rot = tau[3 + k] + t - wxIw[k];
    nu1[k] = fmaf(M.h, lin * M.inv_mass, x.nu[k]);
    nu1[3 + k] = fmaf(M.h, rot * M.inv_inertia[k], x.nu[3 + k]);
  }
  float lnu1[6], LR[3][3], lq[4];
  pose_vjp(M.h, x.q, R, nu1, lx, lnu1, LR, lq);
  float llin[3], lrot[3], lv[3], lw[3], ly[3], lt[3] = {0.f, 0.f, 0.f};
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    llin[k] = M.h * M.inv_mass * lnu1[k];
    lrot[k] = M.h * M.inv_inertia[k] * lnu1[3 + k];
    ltau[k] += llin[k];
    ltau[3 + k] += lrot[k];
    lv[k] = llin[k] * (-2.0f * M.kf_drag[k] * fabsf(v[k]) - M.c_visc_f);
    lw[k] = lrot[k] * (-2.0f * M.kt_drag[k] * fabsf(w[k]) - M.c_visc_t);
    LR[2][k] -= mg * llin[k];
    ly[k] = -m * llin[k];
  }
  cross_vjp(w, v, ly, lw, lv);
#pragma unroll
  for (int k = 0; k < 3; ++k) ly[k] = -lrot[k];
  cross_vjp(w, Iw, ly, lw, lt);
#pragma unroll
  for (int k = 0; k < 3; ++k) lw[k] += M.inertia[k] * lt[k];
  rot_vjp(x.q, LR, lq);
#pragma unroll
  for (int k = 0; k < 4; ++k) lx.q[k] = lq[k];
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lx.nu[k] = lnu1[k] + lv[k];
    lx.nu[3 + k] = lnu1[3 + k] + lw[k];
  }
}

// Save the step's input (x, goal, g, t_ep and the mean of the history rows of
// st) to the step scratch sc [28][n].
__device__ __forceinline__ void paper_save_step(const Model& M, const paper::Env& e,
                                                const float* st, float* sc, size_t n, int i) {
  float mean[6];
  const float inv_k = 1.0f / (float)M.mavg_len;
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    float sum = 0.0f;
    for (int j = 0; j < M.mavg_len; ++j) sum += st[(13 + 6 * j + k) * n + i];
    mean[k] = sum * inv_k;
  }
  const float v[kPScratchF] = {e.p[0], e.p[1], e.p[2], e.q[0], e.q[1], e.q[2], e.q[3],
                               e.nu[0], e.nu[1], e.nu[2], e.nu[3], e.nu[4], e.nu[5],
                               e.pd[0], e.pd[1], e.pd[2], e.qd[0], e.qd[1], e.qd[2], e.qd[3],
                               e.g, __int_as_float(e.t_ep), mean[0], mean[1], mean[2], mean[3],
                               mean[4], mean[5]};
#pragma unroll
  for (int k = 0; k < kPScratchF; ++k) sc[k * n + i] = v[k];
}

__device__ __forceinline__ void paper_load_step(const float* sc, size_t n, int i, paper::Env& e,
                                                int* t_ep, float mean[6]) {
  float v[kPScratchF];
#pragma unroll
  for (int k = 0; k < kPScratchF; ++k) v[k] = sc[k * n + i];
#pragma unroll
  for (int k = 0; k < 3; ++k) { e.p[k] = v[k]; e.pd[k] = v[13 + k]; }
#pragma unroll
  for (int k = 0; k < 4; ++k) { e.q[k] = v[3 + k]; e.qd[k] = v[16 + k]; }
#pragma unroll
  for (int k = 0; k < 6; ++k) { e.nu[k] = v[7 + k]; mean[k] = v[22 + k]; }
  e.g = v[20];
  *t_ep = __float_as_int(v[21]);
}

// Backward of one paper-model control step taken from the input saved in sc
// with actions a: on entry (lx, lh) = dJ/d(post-step state) (the reset cut
// already applied), on exit dJ/d(pre-step state); la = dJ/da (zero where the
// command saturates).
__device__ void paper_step_vjp(const Model& M, const float* sc, size_t n, int i,
                               const float a[paper::kAct], float coef, X& lx,
                               float (&lh)[paper::kHist][6], float la[paper::kAct]) {
  const int K = M.mavg_len;
  const float inv_k = 1.0f / (float)K;
  paper::Env es;
  int t_ep;
  float mean[6];
  paper_load_step(sc, n, i, es, &t_ep, mean);
  float a_c[paper::kAct], tau[6];
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k) a_c[k] = fminf(fmaxf(a[k], -1.0f), 1.0f);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    tau[k] = M.f_max * a_c[k];
    tau[3 + k] = M.tau_max * a_c[3 + k];
  }
  X xs[8];
  for (int s = 0; s < M.substeps; ++s) {
#pragma unroll
    for (int k = 0; k < 3; ++k) xs[s].p[k] = es.p[k];
#pragma unroll
    for (int k = 0; k < 4; ++k) xs[s].q[k] = es.q[k];
#pragma unroll
    for (int k = 0; k < 6; ++k) xs[s].nu[k] = es.nu[k];
    paper::substep(M, es, tau);
  }
  // the history slot written after this step's reward held a_c
  const int slot = t_ep % K;
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    la[k] = lh[slot][k];
    lh[slot][k] = 0.0f;
  }
  // reward on the post-step state
  float o[paper::kObs], lo[paper::kObs];
  paper::observe(es, o);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    lo[k] = -coef * M.w_pos * 2.0f * M.w_axes[k] * M.w_axes[k] * o[k];
    lo[3 + k] = -coef * M.w_att * 2.0f * o[3 + k];
    lo[6 + k] = 0.0f;
    lo[9 + k] = -coef * M.w_vel * 2.0f * o[9 + k];
    la[3 + k] += -coef * M.w_act * 2.0f * a_c[3 + k];
  }
  paper_obs_vjp(es, lo, lx);
#pragma unroll
  for (int k = 0; k < 6; ++k) {
    const float dk = a_c[k] - mean[k];
    la[k] += -coef * M.w_mavg * 2.0f * dk;
    const float lm = coef * M.w_mavg * 2.0f * dk * inv_k;
    for (int j = 0; j < K; ++j) lh[j][k] += lm;
  }
  float ltau[6] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int s = M.substeps - 1; s >= 0; --s) paper_substep_vjp(M, es, xs[s], tau, lx, ltau);
#pragma unroll
  for (int k = 0; k < 3; ++k) {
    la[k] += M.f_max * ltau[k];
    la[3 + k] += M.tau_max * ltau[3 + k];
  }
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k)
    if (!(a[k] >= -1.0f && a[k] <= 1.0f)) la[k] = 0.0f;
}

__global__ void __launch_bounds__(kAdjThreads, 4) k_paper_adjoint(
    const Model M, Buffers B, const float* __restrict__ act, int T,
    const float* __restrict__ coef, const float* __restrict__ lam_T, float* __restrict__ g_act,
    float* __restrict__ lam_0, float* __restrict__ rew, uint8_t* __restrict__ done,
    float* __restrict__ scratch, Status* st) {
  using namespace paper;
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  const uint32_t id = M.id_base + (uint32_t)i;
  float* hsc = scratch + (size_t)T * kPScratchF * n;    // [61][n]: rows 13.. the history
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  for (int r = 13; r < paper::kStateF; ++r) hsc[r * n + i] = B.state[r * n + i];
  uint64_t ends = 0;
  // Step t + 1's actions are loaded while step t integrates (and step t - 1's
  // while the reverse sweep differentiates step t).
  float a_next[paper::kAct];
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k) a_next[k] = T > 0 ? __ldg(act + (size_t)k * n + i) : 0.0f;
  for (int t = 0; t < T; ++t) {
    paper_save_step(M, e, hsc, scratch + (size_t)t * kPScratchF * n, n, i);
    float a[paper::kAct];
#pragma unroll
    for (int k = 0; k < paper::kAct; ++k) a[k] = a_next[k];
    if (t + 1 < T) {
#pragma unroll
      for (int k = 0; k < paper::kAct; ++k)
        a_next[k] = __ldg(act + ((size_t)(t + 1) * paper::kAct + k) * n + i);
    }
    bool d;
    const float r = paper::physics_step(M, id, e, a, paper::hist_rows(hsc, (int)n, i), &d);
    if (d) ends |= 1ull << t;
    if (rew) rew[(size_t)t * n + i] = r;
    if (done) done[(size_t)t * n + i] = d ? 1 : 0;
  }
  X lx;
  float lh[paper::kHist][6];
#pragma unroll
  for (int k = 0; k < kX; ++k) {
    const float v = lam_T ? __ldg(lam_T + k * n + i) : 0.0f;
    if (k < 3) lx.p[k] = v;
    else if (k < 7) lx.q[k - 3] = v;
    else lx.nu[k - 7] = v;
  }
  for (int j = 0; j < paper::kHist; ++j)
#pragma unroll
    for (int k = 0; k < 6; ++k) lh[j][k] = lam_T ? __ldg(lam_T + (13 + 6 * j + k) * n + i) : 0.0f;
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k)
    a_next[k] = T > 0 ? __ldg(act + ((size_t)(T - 1) * paper::kAct + k) * n + i) : 0.0f;
  for (int t = T - 1; t >= 0; --t) {
    if ((ends >> t) & 1ull) {
#pragma unroll
      for (int k = 0; k < 3; ++k) lx.p[k] = 0.f;
#pragma unroll
      for (int k = 0; k < 4; ++k) lx.q[k] = 0.f;
#pragma unroll
      for (int k = 0; k < 6; ++k) lx.nu[k] = 0.f;
      for (int j = 0; j < paper::kHist; ++j)
#pragma unroll
        for (int k = 0; k < 6; ++k) lh[j][k] = 0.f;
    }
    float a[paper::kAct], la[paper::kAct];
#pragma unroll
    for (int k = 0; k < paper::kAct; ++k) a[k] = a_next[k];
    if (t > 0) {
#pragma unroll
      for (int k = 0; k < paper::kAct; ++k)
        a_next[k] = __ldg(act + ((size_t)(t - 1) * paper::kAct + k) * n + i);
    }
    paper_step_vjp(M, scratch + (size_t)t * kPScratchF * n, n, i, a, __ldg(coef + t), lx, lh, la);
#pragma unroll
    for (int k = 0; k < paper::kAct; ++k)
      g_act[((size_t)t * paper::kAct + k) * n + i] = la[k];
  }
  float s = 0.0f;
#pragma unroll
  for (int k = 0; k < 3; ++k) s += lx.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) s += lx.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) s += lx.nu[k];
  if (!isfinite(s)) flag_nan(st, i);
  if (lam_0) {
#pragma unroll
    for (int k = 0; k < 3; ++k) lam_0[k * n + i] = lx.p[k];
#pragma unroll
    for (int k = 0; k < 4; ++k) lam_0[(3 + k) * n + i] = lx.q[k];
#pragma unroll
    for (int k = 0; k < 6; ++k) lam_0[(7 + k) * n + i] = lx.nu[k];
    for (int j = 0; j < paper::kHist; ++j)
#pragma unroll
      for (int k = 0; k < 6; ++k) lam_0[(13 + 6 * j + k) * n + i] = lh[j][k];
  }
}

// ---- SHAC in closed loop on the paper model ----

// Observation row (12 + the constant 1, zeros up to ldx) of each env's state;
// with sc, the step's scratch (its history mean from the env's state rows).
__global__ void __launch_bounds__(kAdjThreads) k_shac_obs_paper(const Model M, Buffers B,
                                                                float* __restrict__ sc,
                                                                float* __restrict__ X, int ldx,
                                                                float* __restrict__ obs_fm,
                                                                int t) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  if (sc) paper_save_step(M, e, B.state, sc, (size_t)M.n, i);
  float o[paper::kObs];
  paper::observe(e, o);
  float* x = X + (size_t)i * ldx;
#pragma unroll
  for (int k = 0; k < paper::kObs; ++k) x[k] = o[k];
  x[paper::kObs] = 1.0f;
  for (int k = paper::kObs + 1; k < ldx; ++k) x[k] = 0.0f;
  if (obs_fm) {
#pragma unroll
    for (int k = 0; k < paper::kObs; ++k) obs_fm[((size_t)t * paper::kObs + k) * M.n + i] = o[k];
  }
}

// a = mu + exp(clamp(ls)) eps for the 6 wrench commands (eps: the first six
// action normals).
__device__ __forceinline__ void paper_shac_action(const Model& M, const float* __restrict__ y,
                                                  const float eps[8], float a[paper::kAct],
                                                  float sig[paper::kAct], bool in[paper::kAct]) {
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k) {
    const float raw = y[paper::kAct + k];
    in[k] = raw >= M.logstd_min && raw <= M.logstd_max;
    sig[k] = expf(fminf(fmaxf(raw, M.logstd_min), M.logstd_max));
    a[k] = fmaf(sig[k], eps[k], y[k]);
  }
}

__global__ void __launch_bounds__(kAdjThreads) k_shac_step_paper(const Model M, Buffers B,
                                                                 const float* __restrict__ Y,
                                                                 int ldy, uint64_t t_g,
                                                                 float* __restrict__ rew,
                                                                 uint8_t* __restrict__ done,
                                                                 Status* st) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  paper::Env e;
  paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  const uint32_t id = M.id_base + (uint32_t)i;
  float eps[8], a[paper::kAct], sig[paper::kAct];
  bool in[paper::kAct];
  action_noise(id, M.seed, t_g, eps);
  paper_shac_action(M, Y + (size_t)i * ldy, eps, a, sig, in);
  bool d;
  const float r = paper::physics_step(M, id, e, a, paper::hist_rows(B.state, M.n, i), &d);
  if (!paper::env_finite(e)) flag_nan(st, i);
  paper::store_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  rew[i] = r;
  done[i] = d ? 1 : 0;
}

// Backward of one closed-loop paper step: lam [61][N] (rows 0..12 the pose
// and velocity, 13.. the history) from post- to pre-step, head gradient gY.
__global__ void __launch_bounds__(kAdjThreads) k_shac_bwd_paper(
    const Model M, const float* __restrict__ sc, const float* __restrict__ Y, int ldy,
    const uint8_t* __restrict__ done, uint64_t t_g, const float* __restrict__ coef,
    float* __restrict__ lam, float* __restrict__ gY) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  const uint32_t id = M.id_base + (uint32_t)i;
  X lx;
  float lh[paper::kHist][6];
  const bool cut = done[i] != 0;
#pragma unroll
  for (int k = 0; k < 3; ++k) lx.p[k] = cut ? 0.f : lam[k * n + i];
#pragma unroll
  for (int k = 0; k < 4; ++k) lx.q[k] = cut ? 0.f : lam[(3 + k) * n + i];
#pragma unroll
  for (int k = 0; k < 6; ++k) lx.nu[k] = cut ? 0.f : lam[(7 + k) * n + i];
  for (int j = 0; j < paper::kHist; ++j)
#pragma unroll
    for (int k = 0; k < 6; ++k) lh[j][k] = cut ? 0.f : lam[(13 + 6 * j + k) * n + i];
  float eps[8], a[paper::kAct], sig[paper::kAct], la[paper::kAct];
  bool in[paper::kAct];
  action_noise(id, M.seed, t_g, eps);
  paper_shac_action(M, Y + (size_t)i * ldy, eps, a, sig, in);
  paper_step_vjp(M, sc, n, i, a, __ldg(coef), lx, lh, la);
  float* g = gY + (size_t)i * ldy;
#pragma unroll
  for (int k = 0; k < paper::kAct; ++k) {
    g[k] = la[k];
    g[paper::kAct + k] = in[k] ? la[k] * sig[k] * eps[k] : 0.0f;
  }
#pragma unroll
  for (int k = 0; k < 3; ++k) lam[k * n + i] = lx.p[k];
#pragma unroll
  for (int k = 0; k < 4; ++k) lam[(3 + k) * n + i] = lx.q[k];
#pragma unroll
  for (int k = 0; k < 6; ++k) lam[(7 + k) * n + i] = lx.nu[k];
  for (int j = 0; j < paper::kHist; ++j)
#pragma unroll
    for (int k = 0; k < 6; ++k) lam[(13 + 6 * j + k) * n + i] = lh[j][k];
}

// lam (rows 0..12) += (d obs / d state)^T gX at the step's input (sc) or at
// the env's current state (sc NULL).
__global__ void __launch_bounds__(kAdjThreads) k_shac_obs_vjp_paper(
    const Model M, Buffers B, const float* __restrict__ sc, const float* __restrict__ gX,
    int ldx, float* __restrict__ lam) {
  const int i = blockIdx.x * kAdjThreads + threadIdx.x;
  if (i >= M.n) return;
  const size_t n = (size_t)M.n;
  paper::Env e;
  if (sc) {
    int t_ep;
    float mean[6];
    paper_load_step(sc, n, i, e, &t_ep, mean);
  } else {
    paper::load_env(M, B.state, B.params, B.t_ep, B.episode, i, e);
  }
  float lo[paper::kObs];
#pragma unroll
  for (int k = 0; k < paper::kObs; ++k) lo[k] = gX[(size_t)i * ldx + k];
  X lx;
  load_lam(lam, n, i, lx);
  paper_obs_vjp(e, lo, lx);
  store_lam(lam, n, i, lx);
}

}  // namespace

size_t adjoint_step_floats(int n) { return (size_t)kScratchF * (size_t)n; }

size_t adjoint_scratch_floats(int n, int T) {
  // Fossen: T steps of 30 floats; paper: T steps of 28 plus a 61-row history copy
  return ((size_t)T * kScratchF + paper::kStateF) * (size_t)n;
}

namespace shac {

static unsigned blocks(int n) { return (n + kAdjThreads - 1) / kAdjThreads; }

cudaError_t launch_obs(const Model& M, const Buffers& B, float* sc, float* X, int ldx,
                       float* obs_fm, int t, cudaStream_t s) {
  if (M.model == 1)
    k_shac_obs_paper<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, sc, X, ldx, obs_fm, t);
  else
    k_shac_obs<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, sc, X, ldx, obs_fm, t);
  return cudaGetLastError();
}

cudaError_t launch_step(const Model& M, const Buffers& B, const float* Y, int ldy, uint64_t t_g,
                        float* rew, uint8_t* done, Status* st, cudaStream_t s) {
  if (M.model == 1)
    k_shac_step_paper<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, Y, ldy, t_g, rew, done, st);
  else
    k_shac_step<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, Y, ldy, t_g, rew, done, st);
  return cudaGetLastError();
}

cudaError_t launch_bwd(const Model& M, const float* sc, const float* Y, int ldy,
                       const uint8_t* done, uint64_t t_g, const float* coef, float* lam,
                       float* gY, cudaStream_t s) {
  if (M.model == 1)
    k_shac_bwd_paper<<<blocks(M.n), kAdjThreads, 0, s>>>(M, sc, Y, ldy, done, t_g, coef, lam, gY);
  else
    k_shac_bwd<<<blocks(M.n), kAdjThreads, 0, s>>>(M, sc, Y, ldy, done, t_g, coef, lam, gY);
  return cudaGetLastError();
}

cudaError_t launch_obs_vjp(const Model& M, const Buffers& B, const float* sc, const float* gX,
                           int ldx, float* lam, cudaStream_t s) {
  if (M.model == 1)
    k_shac_obs_vjp_paper<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, sc, gX, ldx, lam);
  else
    k_shac_obs_vjp<<<blocks(M.n), kAdjThreads, 0, s>>>(M, B, sc, gX, ldx, lam);
  return cudaGetLastError();
}

cudaError_t launch_objective(int n, int T, const float* rew, const float* coef, const float* V,
                             int ldv, float coef_V, float* J, cudaStream_t s) {
  k_shac_objective<<<blocks(n), kAdjThreads, 0, s>>>(n, T, rew, coef, V, ldv, coef_V, J);
  return cudaGetLastError();
}

cudaError_t launch_fill_col(int n, float* buf, int ld, float v, cudaStream_t s) {
  k_fill_col<<<blocks(n), kAdjThreads, 0, s>>>(n, buf, ld, v);
  return cudaGetLastError();
}

}  // namespace shac

cudaError_t launch_adjoint(const Model& M, const Buffers& B, const float* act, int T,
                           const float* coef, const float* lam_T, float* g_act, float* lam_0,
                           float* rew, uint8_t* done, float* scratch, Status* st,
                           cudaStream_t s) {
  if (M.model == 1) {
    k_paper_adjoint<<<(M.n + kAdjThreads - 1) / kAdjThreads, kAdjThreads, 0, s>>>(
        M, B, act, T, coef, lam_T, g_act, lam_0, rew, done, scratch, st);
    return cudaGetLastError();
  }
  k_adjoint<<<(M.n + kAdjThreads - 1) / kAdjThreads, kAdjThreads, 0, s>>>(
      M, B, act, T, coef, lam_T, g_act, lam_0, rew, done, scratch, st);
  return cudaGetLastError();
}

}  // namespace auv
