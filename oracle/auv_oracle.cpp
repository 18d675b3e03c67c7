// auv_oracle.cpp -- TEST INFRASTRUCTURE, not part of the product path.
//
// A plain, slow, single-threaded CPU restatement of the batched AUV rollout
// step of "Fast Policy Learning for 6-DOF Position Control of Underwater
// Vehicles" (arXiv 2512.13359).  Only tests/, __graft_entry__.smoke() and the
// CPU-baseline leg of bench.py may load this file's shared library.  It shares
// no code, header, table or constant generator with the CUDA library under
// paper_2512_13359_gb300/csrc; the two are written independently from the
// same reading of the paper.
//
// Every environment is stepped one after another, every term of the equations
// of motion is written out as a separate vector, and nothing is blocked, fused
// or reordered for speed.  Arithmetic runs in a template scalar R (double for
// parity, float for the precision study); the reset draws are float by
// definition (they must agree bit for bit with any float implementation).
//
// Model (paper §IV-B "Environment Specifications", §IV-D: the vehicle follows
// Fossen's 6-DOF equations of motion), written in the relative-velocity form
// with a constant irrotational current:
//   (M_RB + M_A) nu_dot = tau - C_RB(nu) nu - C_A(nu_r) nu_r - D(nu_r) nu_r
//                         - g(eta) + M_A nu_c_dot
//   nu_r = nu - [v_c; 0],  v_c = R^T V_c,  nu_c_dot = [-(w x v_c); 0]
//   p_dot = R(q) v,  q_dot = 1/2 q (x) (0, w)
// Observation: paper §IV-B1 (error-based, body frame) with the rotation-matrix
// attitude encoding of §V-A3.  Reward: the weighted-norm form of Eqs. (2)-(7).
// Domain randomisation: §IV-C, widened to mass / added-mass / damping scales,
// a buoyancy offset, a centre-of-buoyancy offset and a water current.
// Episodes: §V-A1 (fixed-length episodes with a fresh random reference).
//
// A second model, the paper's own environment (wrench action of Eq. 1,
// inertia-box fluid model, effective gravity, 12-float axis-angle observation,
// five-term reward of Eqs. 2-7), follows the Fossen model below under the
// names paper_* / oracle_paper_*.
//
// Parity pins for every function here live in tests/test_oracle_*.py.

#include <cmath>
#include <cstdint>
#include <cstring>
#include <cstdlib>

namespace {

// ----------------------------------------------------------------------------
// Model description passed in from Python (ctypes mirror in oracle/oracle.py).
// ----------------------------------------------------------------------------
struct OracleModel {
  int32_t n_substeps;     // physics substeps per control step
  int32_t episode_len;    // control steps per episode (time-limit done)
  uint32_t seed;          // second Philox key word
  int32_t dr_enable;      // 1: draw mass/added-mass/damping scales, dB, r_b
  double dt;              // control period [s]
  double mass;            // rigid-body mass [kg]
  double inertia[3];      // principal moments about the CoG [kg m^2]
  double added_mass[6];   // diagonal of M_A
  double damp_lin[6];     // diagonal of D_L
  double damp_quad[6];    // diagonal of D_Q
  double gravity[3];      // world gravity vector g_w [m/s^2]
  double thrust_max;      // thrust per thruster at |a| = 1 [N]
  double alloc[48];       // thruster allocation B, row-major [6][8]
  double w_pos, w_att, w_act, w_vs;   // reward weights
  float init_pos_range;   // initial position  U[-r, r] per axis [m]
  float init_att_range;   // initial roll/pitch/yaw U[-r, r] [rad]
  float goal_pos_range;   // goal position U[-r, r] per axis [m]
  float goal_yaw_range;   // goal yaw U[-r, r] [rad]
  float current_range;    // water current U[-r, r] per world axis [m/s]
  float dr_scale_lo, dr_scale_hi;  // scale factors U[lo, hi]
  float dr_buoy_range;    // buoyancy offset dB U[-r, r] [N]
  float dr_cob_range;     // centre-of-buoyancy offset U[-r, r] per axis [m]
  // policy / value networks
  int32_t hidden;         // hidden width H
  int32_t policy_out;     // 8 (mean only) or 16 (mean and log-std head)
  int32_t mlp_bf16;       // 1: bf16 operands, fp32 accumulation
  int32_t has_value;      // 1: value network present
  float logstd_fixed[8];  // state-independent log-std when policy_out == 8
  float logstd_min, logstd_max;  // clamp of the log-std head
};

constexpr int kObs = 18;
constexpr int kAct = 8;
constexpr int kStateF = 19;   // p(3) q(4) nu(6) nu_prev(6)
constexpr int kParamF = 17;   // p_d(3) q_d(4) s_m s_a s_d dB r_b(3) V_c(3)

// ----------------------------------------------------------------------------
// Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy
// as 1, 2, 3", SC'11): ten rounds of two 32x32->64 multiplies, the Weyl key
// schedule added between rounds.
// ----------------------------------------------------------------------------
void philox4x32_10(const uint32_t ctr_in[4], uint32_t key0, uint32_t key1,
                   uint32_t out[4]) {
  const uint32_t kMul0 = 0xD2511F53u, kMul1 = 0xCD9E8D57u;
  const uint32_t kWeyl0 = 0x9E3779B9u, kWeyl1 = 0xBB67AE85u;
  uint32_t c0 = ctr_in[0], c1 = ctr_in[1], c2 = ctr_in[2], c3 = ctr_in[3];
  uint32_t k0 = key0, k1 = key1;
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += kWeyl0;
      k1 += kWeyl1;
    }
    uint64_t prod0 = (uint64_t)kMul0 * (uint64_t)c0;
    uint64_t prod1 = (uint64_t)kMul1 * (uint64_t)c2;
    uint32_t hi0 = (uint32_t)(prod0 >> 32), lo0 = (uint32_t)prod0;
    uint32_t hi1 = (uint32_t)(prod1 >> 32), lo1 = (uint32_t)prod1;
    uint32_t n0 = hi1 ^ c1 ^ k0;
    uint32_t n1 = lo1;
    uint32_t n2 = hi0 ^ c3 ^ k1;
    uint32_t n3 = lo0;
    c0 = n0; c1 = n1; c2 = n2; c3 = n3;
  }
  out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

// A 32-bit word -> uniform in the open interval (0, 1): the top 23 bits,
// centred in their cell, so every value is exact in float.
float word_to_uniform(uint32_t x) {
  uint32_t odd = (x >> 9) * 2u + 1u;        // 24-bit odd integer
  return (float)odd * 5.9604644775390625e-8f; // 2^-24
}

// Stream layout.  Key = (env id, seed).  Counter word 2 selects the stream:
// 0 = action noise (words 0,1 = global step), 1 = episode reset (words 0,1 =
// episode index).  Word 3 numbers the 4-word blocks within one draw.
void draw_words(uint32_t env_id, uint32_t seed, uint64_t index, uint32_t stream,
                int n_blocks, uint32_t* words) {
  for (int b = 0; b < n_blocks; ++b) {
    uint32_t ctr[4] = {(uint32_t)index, (uint32_t)(index >> 32), stream,
                       (uint32_t)b};
    philox4x32_10(ctr, env_id, seed, words + 4 * b);
  }
}

// Box-Muller transform of uniform pairs (u_even, u_odd) -> two standard
// normals: r = sqrt(-2 ln u_even), angle 2 pi u_odd.
void box_muller8(const float u[8], double eps[8]) {
  const double two_pi = 6.283185307179586476925286766559;
  for (int k = 0; k < 4; ++k) {
    double r = std::sqrt(-2.0 * std::log((double)u[2 * k]));
    double ang = two_pi * (double)u[2 * k + 1];
    eps[2 * k] = r * std::cos(ang);
    eps[2 * k + 1] = r * std::sin(ang);
  }
}

// ----------------------------------------------------------------------------
// Reset draws (float, bit-exact by construction).  Half-angle sine and cosine
// come from fixed-degree Taylor polynomials evaluated by Horner's rule with
// fused multiply-adds in a fixed order, so any IEEE implementation of the same
// steps returns the same bits.
// ----------------------------------------------------------------------------
float taylor_sin(float x) {   // x - x^3/3! + ... - x^15/15!, |x| <= pi/2
  const float x2 = x * x;
  float p = (float)(-1.0 / 1307674368000.0);       // -1/15!
  p = std::fmaf(p, x2, (float)(1.0 / 6227020800.0));   // +1/13!
  p = std::fmaf(p, x2, (float)(-1.0 / 39916800.0));    // -1/11!
  p = std::fmaf(p, x2, (float)(1.0 / 362880.0));       // +1/9!
  p = std::fmaf(p, x2, (float)(-1.0 / 5040.0));        // -1/7!
  p = std::fmaf(p, x2, (float)(1.0 / 120.0));          // +1/5!
  p = std::fmaf(p, x2, (float)(-1.0 / 6.0));           // -1/3!
  p = std::fmaf(p, x2, 1.0f);
  return x * p;
}

float taylor_cos(float x) {   // 1 - x^2/2! + ... + x^16/16!, |x| <= pi/2
  const float x2 = x * x;
  float p = (float)(1.0 / 20922789888000.0);        // +1/16!
  p = std::fmaf(p, x2, (float)(-1.0 / 87178291200.0));  // -1/14!
  p = std::fmaf(p, x2, (float)(1.0 / 479001600.0));     // +1/12!
  p = std::fmaf(p, x2, (float)(-1.0 / 3628800.0));      // -1/10!
  p = std::fmaf(p, x2, (float)(1.0 / 40320.0));         // +1/8!
  p = std::fmaf(p, x2, (float)(-1.0 / 720.0));          // -1/6!
  p = std::fmaf(p, x2, (float)(1.0 / 24.0));            // +1/4!
  p = std::fmaf(p, x2, (float)(-1.0 / 2.0));            // -1/2!
  p = std::fmaf(p, x2, 1.0f);
  return p;
}

// Symmetric range draw U[-r, r] and interval draw U[lo, hi].
float draw_sym(float u, float r) { return std::fmaf(u, r + r, -r); }
float draw_interval(float u, float lo, float hi) {
  return std::fmaf(u, hi - lo, lo);
}

struct ResetDraw {
  float p[3], q[4], p_d[3], q_d[4];
  float s_m, s_a, s_d, dB, r_b[3], V_c[3];
};

// Episode start (§V-A1: a random reference per episode; §IV-C: per-env
// randomised parameters).  Twenty uniforms, in this order: initial position
// x,y,z; roll, pitch, yaw; goal x,y,z; goal yaw; current x,y,z; s_m, s_a,
// s_d; dB; r_b x,y,z.  All twenty are drawn whatever is enabled.
ResetDraw reset_draw(const OracleModel& m, uint32_t env_id, uint32_t episode) {
  uint32_t w[20];
  draw_words(env_id, m.seed, episode, 1u, 5, w);
  float u[20];
  for (int j = 0; j < 20; ++j) u[j] = word_to_uniform(w[j]);
  ResetDraw d;
  for (int k = 0; k < 3; ++k) d.p[k] = draw_sym(u[k], m.init_pos_range);
  float roll = draw_sym(u[3], m.init_att_range);
  float pitch = draw_sym(u[4], m.init_att_range);
  float yaw = draw_sym(u[5], m.init_att_range);
  for (int k = 0; k < 3; ++k) d.p_d[k] = draw_sym(u[6 + k], m.goal_pos_range);
  float goal_yaw = draw_sym(u[9], m.goal_yaw_range);
  for (int k = 0; k < 3; ++k) d.V_c[k] = draw_sym(u[10 + k], m.current_range);
  if (m.dr_enable) {
    d.s_m = draw_interval(u[13], m.dr_scale_lo, m.dr_scale_hi);
    d.s_a = draw_interval(u[14], m.dr_scale_lo, m.dr_scale_hi);
    d.s_d = draw_interval(u[15], m.dr_scale_lo, m.dr_scale_hi);
    d.dB = draw_sym(u[16], m.dr_buoy_range);
    for (int k = 0; k < 3; ++k) d.r_b[k] = draw_sym(u[17 + k], m.dr_cob_range);
  } else {
    d.s_m = d.s_a = d.s_d = 1.0f;
    d.dB = 0.0f;
    d.r_b[0] = d.r_b[1] = d.r_b[2] = 0.0f;
  }
  // Attitude from Z-Y-X Euler angles: q = q_z(yaw) (x) q_y(pitch) (x) q_x(roll).
  float cr = taylor_cos(0.5f * roll), sr = taylor_sin(0.5f * roll);
  float cp = taylor_cos(0.5f * pitch), sp = taylor_sin(0.5f * pitch);
  float cy = taylor_cos(0.5f * yaw), sy = taylor_sin(0.5f * yaw);
  float a = cy * cp, b = sy * sp, c = cy * sp, e = sy * cp;
  d.q[0] = std::fmaf(a, cr, b * sr);
  d.q[1] = std::fmaf(a, sr, -(b * cr));
  d.q[2] = std::fmaf(c, cr, e * sr);
  d.q[3] = std::fmaf(e, cr, -(c * sr));
  // Goal attitude: yaw only.
  d.q_d[0] = taylor_cos(0.5f * goal_yaw);
  d.q_d[1] = 0.0f;
  d.q_d[2] = 0.0f;
  d.q_d[3] = taylor_sin(0.5f * goal_yaw);
  return d;
}

// ----------------------------------------------------------------------------
// Rigid-body kinematics helpers (Hamilton quaternion, body -> world).
// ----------------------------------------------------------------------------
// ----------------------------------------------------------------------------
// Forward-mode automatic differentiation: a dual number v + d e (e^2 = 0)
// carries a value and its derivative along one direction through every
// operation of the templated model code below, so that running the model in
// Dual yields the exact directional derivative of any output (the oracle of
// the adjoint kernels).  Comparisons look at the value only.  The model's
// math calls are unqualified so that double and float keep std:: and Dual
// finds the rules here.
// ----------------------------------------------------------------------------
using std::atan2;
using std::cos;
using std::fabs;
using std::sin;
using std::sqrt;

struct Dual {
  double v, d;
  Dual(double x = 0.0) : v(x), d(0.0) {}
  Dual(double x, double dx) : v(x), d(dx) {}
  explicit operator double() const { return v; }
  explicit operator float() const { return (float)v; }
};
inline Dual operator+(Dual a, Dual b) { return Dual(a.v + b.v, a.d + b.d); }
inline Dual operator-(Dual a, Dual b) { return Dual(a.v - b.v, a.d - b.d); }
inline Dual operator-(Dual a) { return Dual(-a.v, -a.d); }
inline Dual operator*(Dual a, Dual b) { return Dual(a.v * b.v, a.d * b.v + a.v * b.d); }
inline Dual operator/(Dual a, Dual b) {
  return Dual(a.v / b.v, (a.d * b.v - a.v * b.d) / (b.v * b.v));
}
inline Dual& operator+=(Dual& a, Dual b) { return a = a + b; }
inline Dual& operator-=(Dual& a, Dual b) { return a = a - b; }
inline Dual& operator*=(Dual& a, Dual b) { return a = a * b; }
inline Dual& operator/=(Dual& a, Dual b) { return a = a / b; }
inline bool operator<(Dual a, Dual b) { return a.v < b.v; }
inline bool operator>(Dual a, Dual b) { return a.v > b.v; }
inline bool operator<=(Dual a, Dual b) { return a.v <= b.v; }
inline bool operator>=(Dual a, Dual b) { return a.v >= b.v; }
inline bool operator==(Dual a, Dual b) { return a.v == b.v; }
inline bool operator!=(Dual a, Dual b) { return a.v != b.v; }
inline Dual sqrt(Dual a) {
  const double s = std::sqrt(a.v);
  return Dual(s, a.d == 0.0 ? 0.0 : a.d / (2.0 * s));
}
inline Dual fabs(Dual a) { return a.v < 0.0 ? -a : a; }
inline Dual sin(Dual a) { return Dual(std::sin(a.v), std::cos(a.v) * a.d); }
inline Dual cos(Dual a) { return Dual(std::cos(a.v), -std::sin(a.v) * a.d); }
inline Dual atan2(Dual y, Dual x) {
  return Dual(std::atan2(y.v, x.v), (x.v * y.d - y.v * x.d) / (x.v * x.v + y.v * y.v));
}
inline Dual tanh(Dual a) {
  const double t = std::tanh(a.v);
  return Dual(t, (1.0 - t * t) * a.d);
}
inline Dual exp(Dual a) {
  const double e = std::exp(a.v);
  return Dual(e, e * a.d);
}

template <class R>
void quat_to_rot(const R q[4], R Rm[3][3]) {
  R w = q[0], x = q[1], y = q[2], z = q[3];
  Rm[0][0] = 1 - 2 * (y * y + z * z);
  Rm[0][1] = 2 * (x * y - w * z);
  Rm[0][2] = 2 * (x * z + w * y);
  Rm[1][0] = 2 * (x * y + w * z);
  Rm[1][1] = 1 - 2 * (x * x + z * z);
  Rm[1][2] = 2 * (y * z - w * x);
  Rm[2][0] = 2 * (x * z - w * y);
  Rm[2][1] = 2 * (y * z + w * x);
  Rm[2][2] = 1 - 2 * (x * x + y * y);
}

template <class R>
void quat_mul(const R a[4], const R b[4], R out[4]) {
  R w = a[0] * b[0] - a[1] * b[1] - a[2] * b[2] - a[3] * b[3];
  R x = a[0] * b[1] + a[1] * b[0] + a[2] * b[3] - a[3] * b[2];
  R y = a[0] * b[2] - a[1] * b[3] + a[2] * b[0] + a[3] * b[1];
  R z = a[0] * b[3] + a[1] * b[2] - a[2] * b[1] + a[3] * b[0];
  out[0] = w; out[1] = x; out[2] = y; out[3] = z;
}

template <class R>
void cross(const R a[3], const R b[3], R out[3]) {
  R x = a[1] * b[2] - a[2] * b[1];
  R y = a[2] * b[0] - a[0] * b[2];
  R z = a[0] * b[1] - a[1] * b[0];
  out[0] = x; out[1] = y; out[2] = z;
}

template <class R>
void mat_vec(const R M[3][3], const R v[3], R out[3]) {
  for (int i = 0; i < 3; ++i) out[i] = M[i][0] * v[0] + M[i][1] * v[1] + M[i][2] * v[2];
}

template <class R>
void mat_t_vec(const R M[3][3], const R v[3], R out[3]) {
  for (int i = 0; i < 3; ++i) out[i] = M[0][i] * v[0] + M[1][i] * v[1] + M[2][i] * v[2];
}

// ----------------------------------------------------------------------------
// Per-environment state in the oracle's working precision.
// ----------------------------------------------------------------------------
template <class R>
struct Env {
  R p[3], q[4], nu[6], nu_prev[6];
  R p_d[3], q_d[4], s_m, s_a, s_d, dB, r_b[3], V_c[3];
  int32_t t_ep;
  uint32_t episode;
};

template <class R>
void apply_reset(const OracleModel& m, uint32_t env_id, Env<R>& e) {
  ResetDraw d = reset_draw(m, env_id, e.episode);
  for (int k = 0; k < 3; ++k) { e.p[k] = d.p[k]; e.p_d[k] = d.p_d[k]; }
  for (int k = 0; k < 4; ++k) { e.q[k] = d.q[k]; e.q_d[k] = d.q_d[k]; }
  for (int k = 0; k < 6; ++k) { e.nu[k] = 0; e.nu_prev[k] = 0; }
  e.s_m = d.s_m; e.s_a = d.s_a; e.s_d = d.s_d; e.dB = d.dB;
  for (int k = 0; k < 3; ++k) { e.r_b[k] = d.r_b[k]; e.V_c[k] = d.V_c[k]; }
  e.t_ep = 0;
  e.episode += 1u;
}

// nu_dot of the Fossen model above, every term kept separate.
template <class R>
void nu_dot(const OracleModel& m, const Env<R>& e, const R q[4], const R nu[6],
            const R tau[6], R out[6]) {
  R Rm[3][3];
  quat_to_rot(q, Rm);
  const R v[3] = {nu[0], nu[1], nu[2]};
  const R w[3] = {nu[3], nu[4], nu[5]};
  // Randomised inertial and damping parameters.
  const R mass = e.s_m * (R)m.mass;
  const R inertia[3] = {e.s_m * (R)m.inertia[0], e.s_m * (R)m.inertia[1],
                        e.s_m * (R)m.inertia[2]};
  R added[6], dl[6], dq[6];
  for (int k = 0; k < 6; ++k) {
    added[k] = e.s_a * (R)m.added_mass[k];
    dl[k] = e.s_d * (R)m.damp_lin[k];
    dq[k] = e.s_d * (R)m.damp_quad[k];
  }
  // Current in the body frame and relative velocity.
  const R Vc[3] = {e.V_c[0], e.V_c[1], e.V_c[2]};
  R vc[3];
  mat_t_vec(Rm, Vc, vc);
  const R vr[3] = {v[0] - vc[0], v[1] - vc[1], v[2] - vc[2]};
  const R nur[6] = {vr[0], vr[1], vr[2], w[0], w[1], w[2]};
  // Rigid-body Coriolis/centripetal: C_RB(nu) nu = [m (w x v); w x (I w)].
  R crb[6];
  {
    R wxv[3], Iw[3] = {inertia[0] * w[0], inertia[1] * w[1], inertia[2] * w[2]}, wxIw[3];
    cross(w, v, wxv);
    cross(w, Iw, wxIw);
    for (int k = 0; k < 3; ++k) { crb[k] = mass * wxv[k]; crb[3 + k] = wxIw[k]; }
  }
  // Added-mass Coriolis: C_A(nu_r) nu_r = [w x (A1 v_r); v_r x (A1 v_r) + w x (A2 w)].
  R ca[6];
  {
    R A1vr[3] = {added[0] * vr[0], added[1] * vr[1], added[2] * vr[2]};
    R A2w[3] = {added[3] * w[0], added[4] * w[1], added[5] * w[2]};
    R t0[3], t1[3], t2[3];
    cross(w, A1vr, t0);
    cross(vr, A1vr, t1);
    cross(w, A2w, t2);
    for (int k = 0; k < 3; ++k) { ca[k] = t0[k]; ca[3 + k] = t1[k] + t2[k]; }
  }
  // Linear plus quadratic damping on the relative velocity.
  R damp[6];
  for (int k = 0; k < 6; ++k) damp[k] = (dl[k] + dq[k] * fabs(nur[k])) * nur[k];
  // Restoring forces: weight W at the CoG (origin), buoyancy B = W + dB at r_b.
  // With k = R^T g_hat the body-frame gravity direction, the net force is
  // W k - B k = -dB k and the buoyancy moment is r_b x (-B k).
  R rest[6];
  {
    const R g[3] = {(R)m.gravity[0], (R)m.gravity[1], (R)m.gravity[2]};
    const R gnorm = sqrt(g[0] * g[0] + g[1] * g[1] + g[2] * g[2]);
    R kb[3] = {0, 0, 0};
    if (gnorm > 0) {
      const R ghat[3] = {g[0] / gnorm, g[1] / gnorm, g[2] / gnorm};
      mat_t_vec(Rm, ghat, kb);
    }
    const R W = mass * gnorm;
    const R B = W + e.dB;
    const R fb[3] = {-B * kb[0], -B * kb[1], -B * kb[2]};
    R mb[3];
    const R rb[3] = {e.r_b[0], e.r_b[1], e.r_b[2]};
    cross(rb, fb, mb);
    for (int k = 0; k < 3; ++k) { rest[k] = -e.dB * kb[k]; rest[3 + k] = mb[k]; }
  }
  // Current acceleration in the body frame: nu_c_dot = [-(w x v_c); 0].
  R nucdot[6];
  {
    R wxvc[3];
    cross(w, vc, wxvc);
    for (int k = 0; k < 3; ++k) { nucdot[k] = -wxvc[k]; nucdot[3 + k] = 0; }
  }
  // (M_RB + M_A) nu_dot = rhs, M diagonal (CoG at the origin, diagonal M_A).
  const R mrb[6] = {mass, mass, mass, inertia[0], inertia[1], inertia[2]};
  for (int k = 0; k < 6; ++k) {
    R rhs = tau[k] - crb[k] - ca[k] - damp[k] + rest[k] + added[k] * nucdot[k];
    out[k] = rhs / (mrb[k] + added[k]);
  }
}

// Exponential map of a rotation vector phi = h w as a unit quaternion.
template <class R>
void quat_exp(const R phi[3], R dq[4]) {
  R ang = sqrt(phi[0] * phi[0] + phi[1] * phi[1] + phi[2] * phi[2]);
  if (ang == 0) {
    dq[0] = 1; dq[1] = dq[2] = dq[3] = 0;
    return;
  }
  R half = ang / 2;
  R s = sin(half) / ang;
  dq[0] = cos(half);
  dq[1] = s * phi[0]; dq[2] = s * phi[1]; dq[3] = s * phi[2];
}

// One physics substep, semi-implicit (symplectic) Euler: velocity first, then
// position with the new body velocity and attitude by the exponential map of
// the new angular velocity, then renormalisation.
template <class R>
void substep(const OracleModel& m, Env<R>& e, const R tau[6], R h) {
  R acc[6];
  nu_dot(m, e, e.q, e.nu, tau, acc);
  for (int k = 0; k < 6; ++k) e.nu[k] = e.nu[k] + h * acc[k];
  R Rm[3][3];
  quat_to_rot(e.q, Rm);
  R pdot[3];
  const R v[3] = {e.nu[0], e.nu[1], e.nu[2]};
  mat_vec(Rm, v, pdot);
  for (int k = 0; k < 3; ++k) e.p[k] = e.p[k] + h * pdot[k];
  R phi[3] = {h * e.nu[3], h * e.nu[4], h * e.nu[5]};
  R dq[4], qn[4];
  quat_exp(phi, dq);
  quat_mul(e.q, dq, qn);
  R n = sqrt(qn[0] * qn[0] + qn[1] * qn[1] + qn[2] * qn[2] + qn[3] * qn[3]);
  for (int k = 0; k < 4; ++k) e.q[k] = qn[k] / n;
}

// Observation (§IV-B1): body-frame position error, attitude error as the full
// rotation matrix R_e = R(q_d)^T R(q) in column-major order (its first two
// columns are the continuous 6-D encoding), body linear and angular velocity.
template <class R>
void observe(const Env<R>& e, R obs[kObs]) {
  R Rq[3][3], Rd[3][3];
  quat_to_rot(e.q, Rq);
  const R qd[4] = {e.q_d[0], e.q_d[1], e.q_d[2], e.q_d[3]};
  quat_to_rot(qd, Rd);
  const R dp[3] = {e.p[0] - e.p_d[0], e.p[1] - e.p_d[1], e.p[2] - e.p_d[2]};
  R dpb[3];
  mat_t_vec(Rq, dp, dpb);
  R Re[3][3];
  for (int i = 0; i < 3; ++i)
    for (int j = 0; j < 3; ++j)
      Re[i][j] = Rd[0][i] * Rq[0][j] + Rd[1][i] * Rq[1][j] + Rd[2][i] * Rq[2][j];
  obs[0] = dpb[0]; obs[1] = dpb[1]; obs[2] = dpb[2];
  for (int j = 0; j < 3; ++j)
    for (int i = 0; i < 3; ++i) obs[3 + 3 * j + i] = Re[i][j];
  for (int k = 0; k < 6; ++k) obs[12 + k] = e.nu[k];
}

// Geodesic attitude error: the angle of q_e = conj(q_d) (x) q, in [0, pi]
// (the norm of the paper's axis-angle error vector, Eq. (4)).
template <class R>
R attitude_angle(const Env<R>& e) {
  const R qdc[4] = {e.q_d[0], -e.q_d[1], -e.q_d[2], -e.q_d[3]};
  R qe[4];
  quat_mul(qdc, e.q, qe);
  R vn = sqrt(qe[1] * qe[1] + qe[2] * qe[2] + qe[3] * qe[3]);
  return 2 * atan2(vn, fabs(qe[0]));
}

// Reward: -w_pos ||dp|| - w_att theta_e - w_act ||a_c||^2 - w_vs ||nu - nu_prev||^2,
// evaluated on the post-step state.
template <class R>
R reward(const OracleModel& m, const Env<R>& e, const R a_c[kAct]) {
  R d2 = 0;
  for (int k = 0; k < 3; ++k) d2 += (e.p[k] - e.p_d[k]) * (e.p[k] - e.p_d[k]);
  R a2 = 0;
  for (int k = 0; k < kAct; ++k) a2 += a_c[k] * a_c[k];
  R v2 = 0;
  for (int k = 0; k < 6; ++k) v2 += (e.nu[k] - e.nu_prev[k]) * (e.nu[k] - e.nu_prev[k]);
  return -(R)m.w_pos * sqrt(d2) - (R)m.w_att * attitude_angle(e) -
         (R)m.w_act * a2 - (R)m.w_vs * v2;
}

// Thruster allocation: tau = B (thrust_max clip(a, -1, 1)).
template <class R>
void allocate(const OracleModel& m, const R a[kAct], R a_c[kAct], R tau[6]) {
  for (int k = 0; k < kAct; ++k) a_c[k] = a[k] < -1 ? (R)-1 : (a[k] > 1 ? (R)1 : a[k]);
  for (int r = 0; r < 6; ++r) {
    R s = 0;
    for (int k = 0; k < kAct; ++k) s += (R)m.alloc[r * kAct + k] * ((R)m.thrust_max * a_c[k]);
    tau[r] = s;
  }
}

// One control step with the action given.  Returns the reward; sets *done.
template <class R>
R control_step(const OracleModel& m, uint32_t env_id, Env<R>& e, const R a[kAct],
               uint8_t* done) {
  R a_c[kAct], tau[6];
  allocate(m, a, a_c, tau);
  for (int k = 0; k < 6; ++k) e.nu_prev[k] = e.nu[k];
  const R h = (R)m.dt / (R)m.n_substeps;
  for (int s = 0; s < m.n_substeps; ++s) substep(m, e, tau, h);
  R r = reward(m, e, a_c);
  e.t_ep += 1;
  *done = (e.t_ep == m.episode_len) ? 1 : 0;
  if (*done) apply_reset(m, env_id, e);
  return r;
}

// ----------------------------------------------------------------------------
// Policy / value multilayer perceptrons: tanh(W1 x + b1) -> tanh(W2 h + b2) ->
// W3 h + b3, weights stored row-major [out][in] as
// [W1 | b1 | W2 | b2 | W3 | b3].  In bf16 mode the weights, the network input
// and both hidden activations are rounded to bfloat16 (round to nearest even),
// products are accumulated exactly, biases are added in full precision.
// ----------------------------------------------------------------------------
float to_bf16(double x) {
  // Round to the nearest bfloat16 value (8 significant bits, float's exponent
  // range), ties to even: write x = f 2^e with 1/2 <= |f| < 1, round f 2^8 to
  // the nearest integer (ties to even) and scale back.  Powers-of-two scaling
  // is exact, so there is a single rounding.
  if (x == 0 || std::isnan(x) || std::isinf(x)) return (float)x;
  int e = 0;
  double f = std::frexp(x, &e);
  double r = std::nearbyint(std::ldexp(f, 8));
  return (float)std::ldexp(r, e - 8);
}

template <class R>
R round_act(R x, bool bf16) { return bf16 ? (R)to_bf16((double)x) : x; }

template <class R>
void mlp_forward(const float* wts, int in_dim, int hidden, int out_dim, bool bf16,
                 const R* x_in, R* out) {
  const float* W1 = wts;
  const float* b1 = W1 + hidden * in_dim;
  const float* W2 = b1 + hidden;
  const float* b2 = W2 + hidden * hidden;
  const float* W3 = b2 + hidden;
  const float* b3 = W3 + out_dim * hidden;
  auto wq = [&](float w) -> R { return bf16 ? (R)to_bf16((double)w) : (R)w; };
  R* x = new R[in_dim];
  R* h1 = new R[hidden];
  R* h2 = new R[hidden];
  for (int i = 0; i < in_dim; ++i) x[i] = round_act(x_in[i], bf16);
  for (int j = 0; j < hidden; ++j) {
    R s = 0;
    for (int i = 0; i < in_dim; ++i) s += wq(W1[j * in_dim + i]) * x[i];
    h1[j] = round_act((R)std::tanh(s + (R)b1[j]), bf16);
  }
  for (int j = 0; j < hidden; ++j) {
    R s = 0;
    for (int i = 0; i < hidden; ++i) s += wq(W2[j * hidden + i]) * h1[i];
    h2[j] = round_act((R)std::tanh(s + (R)b2[j]), bf16);
  }
  for (int j = 0; j < out_dim; ++j) {
    R s = 0;
    for (int i = 0; i < hidden; ++i) s += wq(W3[j * hidden + i]) * h2[i];
    out[j] = s + (R)b3[j];
  }
  delete[] x; delete[] h1; delete[] h2;
}

// Gaussian policy head: mean and log-std (fixed vector or clamped head output).
template <class R>
void policy_head(const OracleModel& m, const float* pol_w, const R obs[kObs],
                 R mu[kAct], R logstd[kAct]) {
  R out[16];
  mlp_forward<R>(pol_w, kObs, m.hidden, m.policy_out, m.mlp_bf16 != 0, obs, out);
  for (int k = 0; k < kAct; ++k) {
    mu[k] = out[k];
    if (m.policy_out == 16) {
      R ls = out[kAct + k];
      ls = ls < (R)m.logstd_min ? (R)m.logstd_min : ls;
      ls = ls > (R)m.logstd_max ? (R)m.logstd_max : ls;
      logstd[k] = ls;
    } else {
      logstd[k] = (R)m.logstd_fixed[k];
    }
  }
}

// ----------------------------------------------------------------------------
// SoA import / export (state[k*n + i], params[k*n + i]).
// ----------------------------------------------------------------------------
template <class R>
void load_env(const double* st, const double* pr, const int32_t* t_ep,
              const uint32_t* ep, int n, int i, Env<R>& e) {
  for (int k = 0; k < 3; ++k) e.p[k] = (R)st[(0 + k) * n + i];
  for (int k = 0; k < 4; ++k) e.q[k] = (R)st[(3 + k) * n + i];
  for (int k = 0; k < 6; ++k) e.nu[k] = (R)st[(7 + k) * n + i];
  for (int k = 0; k < 6; ++k) e.nu_prev[k] = (R)st[(13 + k) * n + i];
  for (int k = 0; k < 3; ++k) e.p_d[k] = (R)pr[(0 + k) * n + i];
  for (int k = 0; k < 4; ++k) e.q_d[k] = (R)pr[(3 + k) * n + i];
  e.s_m = (R)pr[7 * n + i]; e.s_a = (R)pr[8 * n + i]; e.s_d = (R)pr[9 * n + i];
  e.dB = (R)pr[10 * n + i];
  for (int k = 0; k < 3; ++k) e.r_b[k] = (R)pr[(11 + k) * n + i];
  for (int k = 0; k < 3; ++k) e.V_c[k] = (R)pr[(14 + k) * n + i];
  e.t_ep = t_ep[i];
  e.episode = ep[i];
}

template <class R>
void store_state(const Env<R>& e, int n, int i, double* st) {
  for (int k = 0; k < 3; ++k) st[(0 + k) * n + i] = (double)e.p[k];
  for (int k = 0; k < 4; ++k) st[(3 + k) * n + i] = (double)e.q[k];
  for (int k = 0; k < 6; ++k) st[(7 + k) * n + i] = (double)e.nu[k];
  for (int k = 0; k < 6; ++k) st[(13 + k) * n + i] = (double)e.nu_prev[k];
}

template <class R>
void store_env(const Env<R>& e, int n, int i, double* st, double* pr, int32_t* t_ep,
               uint32_t* ep) {
  store_state(e, n, i, st);
  for (int k = 0; k < 3; ++k) pr[(0 + k) * n + i] = (double)e.p_d[k];
  for (int k = 0; k < 4; ++k) pr[(3 + k) * n + i] = (double)e.q_d[k];
  pr[7 * n + i] = (double)e.s_m; pr[8 * n + i] = (double)e.s_a; pr[9 * n + i] = (double)e.s_d;
  pr[10 * n + i] = (double)e.dB;
  for (int k = 0; k < 3; ++k) pr[(11 + k) * n + i] = (double)e.r_b[k];
  for (int k = 0; k < 3; ++k) pr[(14 + k) * n + i] = (double)e.V_c[k];
  t_ep[i] = e.t_ep;
  ep[i] = e.episode;
}

template <class R>
void replay_impl(const OracleModel& m, int n, const uint32_t* env_ids, double* st,
                 double* pr, int32_t* t_ep, uint32_t* ep, int T, const float* act,
                 double* rew, uint8_t* done, double* trace) {
  for (int i = 0; i < n; ++i) {
    Env<R> e;
    load_env<R>(st, pr, t_ep, ep, n, i, e);
    for (int t = 0; t < T; ++t) {
      R a[kAct];
      for (int k = 0; k < kAct; ++k) a[k] = (R)act[((size_t)t * kAct + k) * n + i];
      uint8_t d;
      R r = control_step(m, env_ids[i], e, a, &d);
      rew[(size_t)t * n + i] = (double)r;
      done[(size_t)t * n + i] = d;
      if (trace) store_state(e, n, i, trace + (size_t)t * kStateF * n);
    }
    store_env(e, n, i, st, pr, t_ep, ep);
  }
}

template <class R>
void rollout_impl(const OracleModel& m, const float* pol_w, const float* val_w, int n,
                  const uint32_t* env_ids, double* st, double* pr, int32_t* t_ep,
                  uint32_t* ep, uint64_t t_g0, int T, double* obs_out, double* act_out,
                  double* logp_out, double* value_out, double* rew_out, uint8_t* done_out) {
  const double half_log_2pi = 0.91893853320467274178032973640562;
  for (int i = 0; i < n; ++i) {
    Env<R> e;
    load_env<R>(st, pr, t_ep, ep, n, i, e);
    for (int t = 0; t < T; ++t) {
      R obs[kObs];
      observe(e, obs);
      R mu[kAct], logstd[kAct];
      policy_head(m, pol_w, obs, mu, logstd);
      uint32_t w[8];
      draw_words(env_ids[i], m.seed, t_g0 + (uint64_t)t, 0u, 2, w);
      float u[8];
      for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
      double eps[8];
      box_muller8(u, eps);
      R a[kAct];
      double logp = 0;
      for (int k = 0; k < kAct; ++k) {
        a[k] = mu[k] + (R)std::exp((double)logstd[k]) * (R)eps[k];
        logp += -0.5 * eps[k] * eps[k] - (double)logstd[k] - half_log_2pi;
      }
      if (value_out && m.has_value) {
        R v;
        mlp_forward<R>(val_w, kObs, m.hidden, 1, m.mlp_bf16 != 0, obs, &v);
        value_out[(size_t)t * n + i] = (double)v;
      }
      if (obs_out)
        for (int k = 0; k < kObs; ++k) obs_out[((size_t)t * kObs + k) * n + i] = (double)obs[k];
      if (act_out)
        for (int k = 0; k < kAct; ++k) act_out[((size_t)t * kAct + k) * n + i] = (double)a[k];
      if (logp_out) logp_out[(size_t)t * n + i] = logp;
      uint8_t d;
      R r = control_step(m, env_ids[i], e, a, &d);
      if (rew_out) rew_out[(size_t)t * n + i] = (double)r;
      if (done_out) done_out[(size_t)t * n + i] = d;
    }
    store_env(e, n, i, st, pr, t_ep, ep);
  }
}

// Classical fourth-order Runge-Kutta on the continuous model with the
// quaternion carried as a 4-vector (q_dot = 1/2 q (x) (0, w)) and renormalised
// only at the end of each step.  Used only as a brute-force reference.
template <class R>
void rk4_deriv(const OracleModel& m, const Env<R>& e, const R y[13], const R tau[6],
               R dy[13]) {
  const R q[4] = {y[3], y[4], y[5], y[6]};
  const R nu[6] = {y[7], y[8], y[9], y[10], y[11], y[12]};
  R Rm[3][3];
  quat_to_rot(q, Rm);
  const R v[3] = {nu[0], nu[1], nu[2]};
  R pd[3];
  mat_vec(Rm, v, pd);
  const R wq[4] = {0, nu[3], nu[4], nu[5]};
  R qd[4];
  quat_mul(q, wq, qd);
  R acc[6];
  nu_dot(m, e, q, nu, tau, acc);
  for (int k = 0; k < 3; ++k) dy[k] = pd[k];
  for (int k = 0; k < 4; ++k) dy[3 + k] = qd[k] / 2;
  for (int k = 0; k < 6; ++k) dy[7 + k] = acc[k];
}

// ============================================================================
// The paper's own environment (§IV-B "Environment Specifications", Eqs. (1)-(7),
// §IV-C), next to the thruster-level Fossen model above:
//  - action: a normalised body wrench a = [F; tau] in [-1, 1]^6, scaled by
//    F_max and tau_max (Eq. 1);
//  - dynamics: a free rigid body (no added mass) in still water under the
//    "inertia" fluid model the paper names: the body is replaced by the
//    uniform box that has its mass and principal moments, and that box feels
//    quadratic pressure drag on its faces and viscous (Stokes) resistance;
//    buoyancy is folded into an effective gravity acting at the centre of
//    mass (centres of gravity and buoyancy coincide), randomised per episode;
//  - observation (12): body-frame position error, axis-angle attitude error,
//    body linear velocity, body angular velocity (§IV-B1);
//  - reward: r_pos + r_att + r_act + r_vel + r_act-mavg (Eqs. 2-7).
// Integration, noise streams and networks are those of the Fossen model.
// ============================================================================
struct PaperModel {
  int32_t n_substeps;     // physics substeps per control step
  int32_t episode_len;    // control steps per episode
  uint32_t seed;          // second Philox key word
  int32_t dr_enable;      // 1: draw the effective gravity offset
  int32_t mavg_len;       // K: actions in the moving average, 1..8
  int32_t pad0;
  double dt;              // control period [s]
  double mass;            // m [kg]
  double inertia[3];      // principal moments about the centre of mass [kg m^2]
  double f_max, tau_max;  // Eq. (1) scaling of the normalised wrench
  double rho;             // fluid density [kg/m^3]
  double visc;            // fluid dynamic viscosity [Pa s]
  double g_eff;           // nominal effective gravity along world -z [m/s^2]
  double w_pos, w_axes[3], w_att, w_act, w_vel, w_mavg;   // Eqs. (2)-(7)
  float goal_pos_range;   // goal position U[-r, r] per axis [m]
  float goal_att_range;   // goal roll, pitch, yaw U[-r, r] [rad]
  float init_pos_range;   // initial position U[-r, r] per axis [m]
  float init_att_range;   // initial roll, pitch, yaw U[-r, r] [rad]
  float dr_gravity_range; // effective gravity offset U[-r, r] [m/s^2]
  int32_t hidden;         // hidden width of both networks
  int32_t policy_out;     // 6 (mean; fixed log-std) or 12 (mean and log-std head)
  int32_t mlp_bf16;
  int32_t has_value;
  float logstd_fixed[6];
  float logstd_min, logstd_max;
};

constexpr int kPObs = 12;
constexpr int kPAct = 6;
constexpr int kPHist = 8;                    // action-history slots kept (K <= 8)
constexpr int kPStateF = 13 + 6 * kPHist;    // p(3) q(4) nu(6) history[8][6]
constexpr int kPParamF = 8;                  // p_d(3) q_d(4) g_eff

template <class R>
struct PaperEnv {
  R p[3], q[4], nu[6], hist[kPHist][6];
  R p_d[3], q_d[4], g_eff;
  int32_t t_ep;
  uint32_t episode;
};

// Z-Y-X Euler angles -> unit quaternion q_z(yaw) (x) q_y(pitch) (x) q_x(roll),
// float, fixed steps (bit-exact across implementations of the same steps).
void euler_to_quat(float roll, float pitch, float yaw, float q[4]) {
  float cr = taylor_cos(0.5f * roll), sr = taylor_sin(0.5f * roll);
  float cp = taylor_cos(0.5f * pitch), sp = taylor_sin(0.5f * pitch);
  float cy = taylor_cos(0.5f * yaw), sy = taylor_sin(0.5f * yaw);
  float a = cy * cp, b = sy * sp, c = cy * sp, e = sy * cp;
  q[0] = std::fmaf(a, cr, b * sr);
  q[1] = std::fmaf(a, sr, -(b * cr));
  q[2] = std::fmaf(c, cr, e * sr);
  q[3] = std::fmaf(e, cr, -(c * sr));
}

// Episode start (§V-A1: a random 6-DOF reference per episode, §IV-C: the
// effective gravity redrawn per environment).  Thirteen uniforms from the
// reset stream, in this order: goal x, y, z; goal roll, pitch, yaw; gravity
// offset; initial x, y, z; initial roll, pitch, yaw.  Velocities and the
// action history start at zero.
template <class R>
void paper_apply_reset(const PaperModel& m, uint32_t env_id, PaperEnv<R>& e) {
  uint32_t w[16];
  draw_words(env_id, m.seed, e.episode, 1u, 4, w);
  float u[13];
  for (int j = 0; j < 13; ++j) u[j] = word_to_uniform(w[j]);
  float qd[4], q0[4];
  euler_to_quat(draw_sym(u[3], m.goal_att_range), draw_sym(u[4], m.goal_att_range),
                draw_sym(u[5], m.goal_att_range), qd);
  euler_to_quat(draw_sym(u[10], m.init_att_range), draw_sym(u[11], m.init_att_range),
                draw_sym(u[12], m.init_att_range), q0);
  for (int k = 0; k < 3; ++k) {
    e.p_d[k] = draw_sym(u[k], m.goal_pos_range);
    e.p[k] = draw_sym(u[7 + k], m.init_pos_range);
  }
  for (int k = 0; k < 4; ++k) { e.q_d[k] = qd[k]; e.q[k] = q0[k]; }
  const float g0 = (float)m.g_eff;
  e.g_eff = m.dr_enable ? g0 + draw_sym(u[6], m.dr_gravity_range) : g0;
  for (int k = 0; k < 6; ++k) e.nu[k] = 0;
  for (int j = 0; j < kPHist; ++j)
    for (int k = 0; k < 6; ++k) e.hist[j][k] = 0;
  e.t_ep = 0;
  e.episode += 1u;
}

// Sides of the uniform box with the body's mass and principal moments:
// I_x = m (b_y^2 + b_z^2) / 12 and so on, solved for the sides.
template <class R>
void paper_box(const PaperModel& m, R b[3]) {
  const R I0 = (R)m.inertia[0], I1 = (R)m.inertia[1], I2 = (R)m.inertia[2], M = (R)m.mass;
  b[0] = sqrt(6 * (I1 + I2 - I0) / M);
  b[1] = sqrt(6 * (I0 + I2 - I1) / M);
  b[2] = sqrt(6 * (I0 + I1 - I2) / M);
}

// Hydrodynamic wrench on the box moving with body velocity nu in still water,
// every term kept separate: pressure drag -1/2 rho A_i |v_i| v_i on the face
// areas A = (b_y b_z, b_x b_z, b_x b_y); its rotational counterpart
// -rho/64 b_i (b_j^4 + b_k^4) |w_i| w_i (the pressure on the halves of the
// faces moving into the fluid, integrated over the face); Stokes resistance
// -3 pi mu d v and -pi mu d^3 w of the sphere of diameter d = (b_x+b_y+b_z)/3.
template <class R>
void paper_fluid(const PaperModel& m, const R nu[6], R f[6]) {
  R b[3];
  paper_box(m, b);
  const R rho = (R)m.rho, mu = (R)m.visc, pi = (R)3.14159265358979323846;
  const R d = (b[0] + b[1] + b[2]) / 3;
  const R area[3] = {b[1] * b[2], b[0] * b[2], b[0] * b[1]};
  for (int k = 0; k < 3; ++k) {
    const int j = (k + 1) % 3, l = (k + 2) % 3;
    const R v = nu[k], w = nu[3 + k];
    const R drag_f = -(R)0.5 * rho * area[k] * fabs(v) * v;
    const R visc_f = -3 * pi * mu * d * v;
    const R b4 = b[j] * b[j] * b[j] * b[j] + b[l] * b[l] * b[l] * b[l];
    const R drag_t = -rho / 64 * b[k] * b4 * fabs(w) * w;
    const R visc_t = -pi * mu * d * d * d * w;
    f[k] = drag_f + visc_f;
    f[3 + k] = drag_t + visc_t;
  }
}

// nu_dot = M_RB^{-1} (tau + fluid(nu) + R^T (0, 0, -m g_eff) - C_RB(nu) nu).
template <class R>
void paper_nu_dot(const PaperModel& m, const PaperEnv<R>& e, const R q[4], const R nu[6],
                  const R tau[6], R out[6]) {
  R Rm[3][3];
  quat_to_rot(q, Rm);
  const R v[3] = {nu[0], nu[1], nu[2]};
  const R w[3] = {nu[3], nu[4], nu[5]};
  const R M = (R)m.mass;
  const R I[3] = {(R)m.inertia[0], (R)m.inertia[1], (R)m.inertia[2]};
  R fl[6];
  paper_fluid(m, nu, fl);
  const R gw[3] = {0, 0, -M * e.g_eff};
  R gb[3];
  mat_t_vec(Rm, gw, gb);
  R wxv[3], Iw[3] = {I[0] * w[0], I[1] * w[1], I[2] * w[2]}, wxIw[3];
  cross(w, v, wxv);
  cross(w, Iw, wxIw);
  for (int k = 0; k < 3; ++k) {
    out[k] = (tau[k] + fl[k] + gb[k] - M * wxv[k]) / M;
    out[3 + k] = (tau[3 + k] + fl[3 + k] - wxIw[k]) / I[k];
  }
}

// One semi-implicit Euler substep (the integrator of the Fossen model).
template <class R>
void paper_substep(const PaperModel& m, PaperEnv<R>& e, const R tau[6], R h) {
  R acc[6];
  paper_nu_dot(m, e, e.q, e.nu, tau, acc);
  for (int k = 0; k < 6; ++k) e.nu[k] = e.nu[k] + h * acc[k];
  R Rm[3][3];
  quat_to_rot(e.q, Rm);
  R pdot[3];
  const R v[3] = {e.nu[0], e.nu[1], e.nu[2]};
  mat_vec(Rm, v, pdot);
  for (int k = 0; k < 3; ++k) e.p[k] = e.p[k] + h * pdot[k];
  R phi[3] = {h * e.nu[3], h * e.nu[4], h * e.nu[5]};
  R dq[4], qn[4];
  quat_exp(phi, dq);
  quat_mul(e.q, dq, qn);
  R n = sqrt(qn[0] * qn[0] + qn[1] * qn[1] + qn[2] * qn[2] + qn[3] * qn[3]);
  for (int k = 0; k < 4; ++k) e.q[k] = qn[k] / n;
}

// Axis-angle vector of q_e = conj(q_d) (x) q (the attitude of the body in the
// goal frame), on the short way round: angle in [0, pi].
template <class R>
void paper_att_error(const PaperEnv<R>& e, R out[3]) {
  const R qdc[4] = {e.q_d[0], -e.q_d[1], -e.q_d[2], -e.q_d[3]};
  R qe[4];
  quat_mul(qdc, e.q, qe);
  if (qe[0] < 0)
    for (int k = 0; k < 4; ++k) qe[k] = -qe[k];
  const R vn = sqrt(qe[1] * qe[1] + qe[2] * qe[2] + qe[3] * qe[3]);
  const R s = vn > 0 ? 2 * atan2(vn, qe[0]) / vn : 2 / qe[0];
  for (int k = 0; k < 3; ++k) out[k] = s * qe[1 + k];
}

// Observation (§IV-B1): [R^T (p - p_d), axis-angle error, v, w].
template <class R>
void paper_observe(const PaperEnv<R>& e, R obs[kPObs]) {
  R Rm[3][3];
  quat_to_rot(e.q, Rm);
  const R dp[3] = {e.p[0] - e.p_d[0], e.p[1] - e.p_d[1], e.p[2] - e.p_d[2]};
  R dpb[3], th[3];
  mat_t_vec(Rm, dp, dpb);
  paper_att_error(e, th);
  for (int k = 0; k < 3; ++k) { obs[k] = dpb[k]; obs[3 + k] = th[k]; }
  for (int k = 0; k < 6; ++k) obs[6 + k] = e.nu[k];
}

// Reward (Eqs. 2-7) on the post-step state with the clipped action a_c and
// the mean of the K previous clipped actions (zeros before the episode's
// K-th step).
template <class R>
R paper_reward(const PaperModel& m, const PaperEnv<R>& e, const R a_c[kPAct]) {
  R obs[kPObs];
  paper_observe(e, obs);
  R r_pos = 0, r_att = 0, r_act = 0, r_vel = 0, r_mavg = 0;
  for (int k = 0; k < 3; ++k) {
    const R dk = (R)m.w_axes[k] * obs[k];
    r_pos += dk * dk;
    r_att += obs[3 + k] * obs[3 + k];
    r_act += a_c[3 + k] * a_c[3 + k];
    r_vel += e.nu[3 + k] * e.nu[3 + k];
  }
  for (int k = 0; k < kPAct; ++k) {
    R mean = 0;
    for (int j = 0; j < m.mavg_len; ++j) mean += e.hist[j][k];
    mean = mean / (R)m.mavg_len;
    r_mavg += (a_c[k] - mean) * (a_c[k] - mean);
  }
  return -(R)m.w_pos * r_pos - (R)m.w_att * r_att - (R)m.w_act * r_act - (R)m.w_vel * r_vel -
         (R)m.w_mavg * r_mavg;
}

// Eq. (1): clip to [-1, 1], scale forces by F_max and torques by tau_max.
template <class R>
void paper_wrench(const PaperModel& m, const R a[kPAct], R a_c[kPAct], R tau[6]) {
  for (int k = 0; k < kPAct; ++k) a_c[k] = a[k] < -1 ? (R)-1 : (a[k] > 1 ? (R)1 : a[k]);
  for (int k = 0; k < 3; ++k) {
    tau[k] = (R)m.f_max * a_c[k];
    tau[3 + k] = (R)m.tau_max * a_c[3 + k];
  }
}

template <class R>
R paper_control_step(const PaperModel& m, uint32_t env_id, PaperEnv<R>& e, const R a[kPAct],
                     uint8_t* done) {
  R a_c[kPAct], tau[6];
  paper_wrench(m, a, a_c, tau);
  const R h = (R)m.dt / (R)m.n_substeps;
  for (int s = 0; s < m.n_substeps; ++s) paper_substep(m, e, tau, h);
  R r = paper_reward(m, e, a_c);
  for (int k = 0; k < kPAct; ++k) e.hist[e.t_ep % m.mavg_len][k] = a_c[k];
  e.t_ep += 1;
  *done = (e.t_ep == m.episode_len) ? 1 : 0;
  if (*done) paper_apply_reset(m, env_id, e);
  return r;
}

template <class R>
void paper_load(const double* st, const double* pr, const int32_t* t_ep, const uint32_t* ep,
                int n, int i, PaperEnv<R>& e) {
  for (int k = 0; k < 3; ++k) e.p[k] = (R)st[k * n + i];
  for (int k = 0; k < 4; ++k) e.q[k] = (R)st[(3 + k) * n + i];
  for (int k = 0; k < 6; ++k) e.nu[k] = (R)st[(7 + k) * n + i];
  for (int j = 0; j < kPHist; ++j)
    for (int k = 0; k < 6; ++k) e.hist[j][k] = (R)st[(13 + 6 * j + k) * n + i];
  for (int k = 0; k < 3; ++k) e.p_d[k] = (R)pr[k * n + i];
  for (int k = 0; k < 4; ++k) e.q_d[k] = (R)pr[(3 + k) * n + i];
  e.g_eff = (R)pr[7 * n + i];
  e.t_ep = t_ep[i];
  e.episode = ep[i];
}

template <class R>
void paper_store_state(const PaperEnv<R>& e, int n, int i, double* st) {
  for (int k = 0; k < 3; ++k) st[k * n + i] = (double)e.p[k];
  for (int k = 0; k < 4; ++k) st[(3 + k) * n + i] = (double)e.q[k];
  for (int k = 0; k < 6; ++k) st[(7 + k) * n + i] = (double)e.nu[k];
  for (int j = 0; j < kPHist; ++j)
    for (int k = 0; k < 6; ++k) st[(13 + 6 * j + k) * n + i] = (double)e.hist[j][k];
}

template <class R>
void paper_store(const PaperEnv<R>& e, int n, int i, double* st, double* pr, int32_t* t_ep,
                 uint32_t* ep) {
  paper_store_state(e, n, i, st);
  for (int k = 0; k < 3; ++k) pr[k * n + i] = (double)e.p_d[k];
  for (int k = 0; k < 4; ++k) pr[(3 + k) * n + i] = (double)e.q_d[k];
  pr[7 * n + i] = (double)e.g_eff;
  t_ep[i] = e.t_ep;
  ep[i] = e.episode;
}

template <class R>
void paper_replay_impl(const PaperModel& m, int n, const uint32_t* env_ids, double* st,
                       double* pr, int32_t* t_ep, uint32_t* ep, int T, const float* act,
                       double* rew, uint8_t* done, double* trace) {
  for (int i = 0; i < n; ++i) {
    PaperEnv<R> e;
    paper_load<R>(st, pr, t_ep, ep, n, i, e);
    for (int t = 0; t < T; ++t) {
      R a[kPAct];
      for (int k = 0; k < kPAct; ++k) a[k] = (R)act[((size_t)t * kPAct + k) * n + i];
      uint8_t d;
      R r = paper_control_step(m, env_ids[i], e, a, &d);
      rew[(size_t)t * n + i] = (double)r;
      done[(size_t)t * n + i] = d;
      if (trace) paper_store_state(e, n, i, trace + (size_t)t * kPStateF * n);
    }
    paper_store(e, n, i, st, pr, t_ep, ep);
  }
}

template <class R>
void paper_rollout_impl(const PaperModel& m, const float* pol_w, const float* val_w, int n,
                        const uint32_t* env_ids, double* st, double* pr, int32_t* t_ep,
                        uint32_t* ep, uint64_t t_g0, int T, double* obs_out, double* act_out,
                        double* logp_out, double* value_out, double* rew_out,
                        uint8_t* done_out) {
  const double half_log_2pi = 0.91893853320467274178032973640562;
  for (int i = 0; i < n; ++i) {
    PaperEnv<R> e;
    paper_load<R>(st, pr, t_ep, ep, n, i, e);
    for (int t = 0; t < T; ++t) {
      R obs[kPObs];
      paper_observe(e, obs);
      R out[12];
      mlp_forward<R>(pol_w, kPObs, m.hidden, m.policy_out, m.mlp_bf16 != 0, obs, out);
      R mu[kPAct], logstd[kPAct];
      for (int k = 0; k < kPAct; ++k) {
        mu[k] = out[k];
        if (m.policy_out == 12) {
          R ls = out[kPAct + k];
          ls = ls < (R)m.logstd_min ? (R)m.logstd_min : ls;
          logstd[k] = ls > (R)m.logstd_max ? (R)m.logstd_max : ls;
        } else {
          logstd[k] = (R)m.logstd_fixed[k];
        }
      }
      // the first six of the eight normals of the action-noise stream
      uint32_t w[8];
      draw_words(env_ids[i], m.seed, t_g0 + (uint64_t)t, 0u, 2, w);
      float u[8];
      for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
      double eps[8];
      box_muller8(u, eps);
      R a[kPAct];
      double logp = 0;
      for (int k = 0; k < kPAct; ++k) {
        a[k] = mu[k] + (R)std::exp((double)logstd[k]) * (R)eps[k];
        logp += -0.5 * eps[k] * eps[k] - (double)logstd[k] - half_log_2pi;
      }
      if (value_out && m.has_value) {
        R v;
        mlp_forward<R>(val_w, kPObs, m.hidden, 1, m.mlp_bf16 != 0, obs, &v);
        value_out[(size_t)t * n + i] = (double)v;
      }
      if (obs_out)
        for (int k = 0; k < kPObs; ++k) obs_out[((size_t)t * kPObs + k) * n + i] = (double)obs[k];
      if (act_out)
        for (int k = 0; k < kPAct; ++k) act_out[((size_t)t * kPAct + k) * n + i] = (double)a[k];
      if (logp_out) logp_out[(size_t)t * n + i] = logp;
      uint8_t d;
      R r = paper_control_step(m, env_ids[i], e, a, &d);
      if (rew_out) rew_out[(size_t)t * n + i] = (double)r;
      if (done_out) done_out[(size_t)t * n + i] = d;
    }
    paper_store(e, n, i, st, pr, t_ep, ep);
  }
}

template <class R>
void paper_rk4_deriv(const PaperModel& m, const PaperEnv<R>& e, const R y[13], const R tau[6],
                     R dy[13]) {
  const R q[4] = {y[3], y[4], y[5], y[6]};
  const R nu[6] = {y[7], y[8], y[9], y[10], y[11], y[12]};
  R Rm[3][3];
  quat_to_rot(q, Rm);
  const R v[3] = {nu[0], nu[1], nu[2]};
  R pd[3];
  mat_vec(Rm, v, pd);
  const R wq[4] = {0, nu[3], nu[4], nu[5]};
  R qd[4];
  quat_mul(q, wq, qd);
  R acc[6];
  paper_nu_dot(m, e, q, nu, tau, acc);
  for (int k = 0; k < 3; ++k) dy[k] = pd[k];
  for (int k = 0; k < 4; ++k) dy[3 + k] = qd[k] / 2;
  for (int k = 0; k < 6; ++k) dy[7 + k] = acc[k];
}


// ----------------------------------------------------------------------------
// Minibatch permutation of the PPO learner: a bijection on [0, M) for each
// epoch, by a balanced four-round Feistel network (Luby & Rackoff 1988) on a
// domain of 2^b >= M codes (b even, b >= 2), walked until it lands in [0, M)
// ("cycle walking", Black & Rogaway 2002).  The round function is Philox4x32-10
// with counter (right half, round, epoch low, epoch high) and key (seed low,
// seed high); its first word, masked to b/2 bits, is the round value.
// ----------------------------------------------------------------------------
int perm_half_bits(uint64_t m) {
  int b = 2;
  while ((1ull << b) < m) b += 2;
  return b / 2;
}

uint32_t feistel_encode(uint32_t x, int h, uint64_t seed, uint64_t epoch) {
  const uint32_t mask = (h >= 32) ? 0xFFFFFFFFu : ((1u << h) - 1u);
  uint32_t left = x >> h, right = x & mask;
  for (uint32_t r = 0; r < 4; ++r) {
    const uint32_t ctr[4] = {right, r, (uint32_t)epoch, (uint32_t)(epoch >> 32)};
    uint32_t out[4];
    philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32), out);
    const uint32_t next_right = left ^ (out[0] & mask);
    left = right;
    right = next_right;
  }
  return (left << h) | right;
}

uint32_t feistel_decode(uint32_t y, int h, uint64_t seed, uint64_t epoch) {
  const uint32_t mask = (h >= 32) ? 0xFFFFFFFFu : ((1u << h) - 1u);
  uint32_t left = y >> h, right = y & mask;
  for (int r = 3; r >= 0; --r) {
    // undo (L, R) -> (R, L ^ F_r(R)): the old right half is the new left
    const uint32_t ctr[4] = {left, (uint32_t)r, (uint32_t)epoch, (uint32_t)(epoch >> 32)};
    uint32_t out[4];
    philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32), out);
    const uint32_t old_left = right ^ (out[0] & mask);
    right = left;
    left = old_left;
  }
  return (left << h) | right;
}

uint32_t minibatch_index(uint32_t j, uint32_t m, uint64_t seed, uint64_t epoch) {
  const int h = perm_half_bits(m);
  uint32_t x = feistel_encode(j, h, seed, epoch);
  while (x >= m) x = feistel_encode(x, h, seed, epoch);
  return x;
}
}  // namespace

extern "C" {

int oracle_abi_version() { return 1; }
int oracle_model_size() { return (int)sizeof(OracleModel); }

void oracle_philox(uint32_t key0, uint32_t key1, const uint32_t* ctr, uint32_t* out) {
  philox4x32_10(ctr, key0, key1, out);
}

// Positions start .. start+count-1 of epoch `epoch`'s permutation of [0, m).
void oracle_minibatch_perm(uint64_t seed, uint64_t epoch, uint32_t m, uint32_t start,
                           uint32_t count, uint32_t* out) {
  for (uint32_t k = 0; k < count; ++k) out[k] = minibatch_index(start + k, m, seed, epoch);
}

// Replay-buffer sample indices: draw `draw`, sample b takes the first word
// of Philox4x32-10 at counter (b, 0x52420000, draw low, draw high) and key
// (seed low, seed high) and maps it to [0, size) by the multiply-high
// floor(word * size / 2^32).
void oracle_rbuf_indices(uint64_t seed, uint64_t draw, uint32_t size, uint32_t count,
                         uint32_t* out) {
  for (uint32_t b = 0; b < count; ++b) {
    const uint32_t ctr[4] = {b, 0x52420000u, (uint32_t)draw, (uint32_t)(draw >> 32)};
    uint32_t w[4];
    philox4x32_10(ctr, (uint32_t)seed, (uint32_t)(seed >> 32), w);
    out[b] = (uint32_t)(((uint64_t)w[0] * (uint64_t)size) >> 32);
  }
}

// One Feistel pass (no cycle walking) forward or back, for the pins.
uint32_t oracle_feistel(uint32_t x, uint32_t m, uint64_t seed, uint64_t epoch, int inverse) {
  const int h = perm_half_bits(m);
  return inverse ? feistel_decode(x, h, seed, epoch) : feistel_encode(x, h, seed, epoch);
}

float oracle_word_to_uniform(uint32_t x) { return word_to_uniform(x); }
float oracle_taylor_sin(float x) { return taylor_sin(x); }
float oracle_taylor_cos(float x) { return taylor_cos(x); }
float oracle_to_bf16(double x) { return to_bf16(x); }

// Action-noise normals for one env at one global step.
void oracle_normals(uint32_t env_id, uint32_t seed, uint64_t t_g, double* eps8) {
  uint32_t w[8];
  draw_words(env_id, seed, t_g, 0u, 2, w);
  float u[8];
  for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
  box_muller8(u, eps8);
}

// Reset every listed env at its current episode index; writes state/params and
// increments the episode index, zeroes t_ep.
void oracle_reset(const OracleModel* m, int n, const uint32_t* env_ids, double* st,
                  double* pr, int32_t* t_ep, uint32_t* ep) {
  for (int i = 0; i < n; ++i) {
    Env<double> e;
    std::memset(&e, 0, sizeof(e));
    e.episode = ep[i];
    apply_reset(*m, env_ids[i], e);
    store_env(e, n, i, st, pr, t_ep, ep);
  }
}

void oracle_replay(const OracleModel* m, int precision, int n, const uint32_t* env_ids,
                   double* st, double* pr, int32_t* t_ep, uint32_t* ep, int T,
                   const float* act, double* rew, uint8_t* done, double* trace) {
  if (precision == 1)
    replay_impl<float>(*m, n, env_ids, st, pr, t_ep, ep, T, act, rew, done, trace);
  else
    replay_impl<double>(*m, n, env_ids, st, pr, t_ep, ep, T, act, rew, done, trace);
}

// Action-replay window objective J = sum_t coef[t] r_t + sum_k lam_T[k] x_T[k]
// (x = p, q, nu after the last step; lam_T may be NULL) from the batch's
// state, and its directional derivative along (dir_s0 on x_0 = p, q, nu;
// dir_act on the actions), computed in Dual.  The batch is not modified.
void oracle_adjoint_window(const OracleModel* m, int n, const uint32_t* env_ids,
                           const double* st, const double* pr, const int32_t* t_ep,
                           const uint32_t* ep, int T, const double* act, const double* coef,
                           const double* lam_T, const double* dir_s0, const double* dir_act,
                           double* J, double* dJ) {
  for (int i = 0; i < n; ++i) {
    Env<Dual> e;
    load_env<Dual>(st, pr, t_ep, ep, n, i, e);
    for (int k = 0; k < 3; ++k) e.p[k].d = dir_s0[(0 + k) * n + i];
    for (int k = 0; k < 4; ++k) e.q[k].d = dir_s0[(3 + k) * n + i];
    for (int k = 0; k < 6; ++k) e.nu[k].d = dir_s0[(7 + k) * n + i];
    Dual obj = 0.0;
    for (int t = 0; t < T; ++t) {
      Dual a[kAct];
      for (int k = 0; k < kAct; ++k) {
        const size_t o = ((size_t)t * kAct + k) * n + i;
        a[k] = Dual(act[o], dir_act[o]);
      }
      uint8_t d;
      obj += Dual(coef[t]) * control_step(*m, env_ids[i], e, a, &d);
    }
    if (lam_T) {
      for (int k = 0; k < 3; ++k) obj += Dual(lam_T[(0 + k) * n + i]) * e.p[k];
      for (int k = 0; k < 4; ++k) obj += Dual(lam_T[(3 + k) * n + i]) * e.q[k];
      for (int k = 0; k < 6; ++k) obj += Dual(lam_T[(7 + k) * n + i]) * e.nu[k];
    }
    J[i] = obj.v;
    dJ[i] = obj.d;
  }
}

// The MLP of the rollout with its weights as dual numbers: values w (float,
// the flat [W1 | b1 | W2 | b2 | W3 | b3] layout) and tangents dw (NULL for 0).
void mlp_dual(const float* w, const double* dw, int in_dim, int hidden, int out_dim,
              const Dual* x, Dual* out) {
  auto W = [&](size_t k) { return Dual((double)w[k], dw ? dw[k] : 0.0); };
  const size_t oW1 = 0, ob1 = oW1 + (size_t)hidden * in_dim, oW2 = ob1 + hidden,
               ob2 = oW2 + (size_t)hidden * hidden, oW3 = ob2 + hidden,
               ob3 = oW3 + (size_t)out_dim * hidden;
  Dual* h1 = new Dual[hidden];
  Dual* h2 = new Dual[hidden];
  for (int j = 0; j < hidden; ++j) {
    Dual s = 0.0;
    for (int i = 0; i < in_dim; ++i) s += W(oW1 + (size_t)j * in_dim + i) * x[i];
    h1[j] = tanh(s + W(ob1 + j));
  }
  for (int j = 0; j < hidden; ++j) {
    Dual s = 0.0;
    for (int i = 0; i < hidden; ++i) s += W(oW2 + (size_t)j * hidden + i) * h1[i];
    h2[j] = tanh(s + W(ob2 + j));
  }
  for (int j = 0; j < out_dim; ++j) {
    Dual s = 0.0;
    for (int i = 0; i < hidden; ++i) s += W(oW3 + (size_t)j * hidden + i) * h2[i];
    out[j] = s + W(ob3 + j);
  }
  delete[] h1;
  delete[] h2;
}

// SHAC's window objective of each env in closed loop (paper §III-A; Xu et al.
// 2022): from the batch's state, T control steps with the reparameterised
// Gaussian policy a = mu(o) + exp(clamp(ls(o))) eps (eps: the rollout's
// action noise at global step t_g0 + t; policy head 2 x 8), then
//   J = sum_t coef[t] r_t + coef_V V(o_T)
// (value network at the observation after the last step; none if val_w is
// NULL).  Returns J and its directional derivative along the policy-weight
// direction dpol, in forward-mode dual numbers.  The batch is not modified.
void oracle_shac_window(const OracleModel* m, const float* pol_w, const double* dpol,
                        const float* val_w, int n, const uint32_t* env_ids, const double* st,
                        const double* pr, const int32_t* t_ep, const uint32_t* ep,
                        uint64_t t_g0, int T, const double* coef, double coef_V, double* J,
                        double* dJ) {
  for (int i = 0; i < n; ++i) {
    Env<Dual> e;
    load_env<Dual>(st, pr, t_ep, ep, n, i, e);
    Dual obj = 0.0;
    for (int t = 0; t < T; ++t) {
      Dual o[kObs], y[2 * kAct], a[kAct];
      observe(e, o);
      mlp_dual(pol_w, dpol, kObs, m->hidden, 2 * kAct, o, y);
      double eps[8];
      uint32_t w[8];
      draw_words(env_ids[i], m->seed, t_g0 + (uint64_t)t, 0u, 2, w);
      float u[8];
      for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
      box_muller8(u, eps);
      for (int k = 0; k < kAct; ++k) {
        Dual ls = y[kAct + k];
        if (ls < Dual(m->logstd_min)) ls = Dual(m->logstd_min);
        if (ls > Dual(m->logstd_max)) ls = Dual(m->logstd_max);
        a[k] = y[k] + exp(ls) * Dual(eps[k]);
      }
      uint8_t d;
      obj += Dual(coef[t]) * control_step(*m, env_ids[i], e, a, &d);
    }
    if (val_w) {
      Dual o[kObs], v[1];
      observe(e, o);
      mlp_dual(val_w, nullptr, kObs, m->hidden, 1, o, v);
      obj += Dual(coef_V) * v[0];
    }
    J[i] = obj.v;
    dJ[i] = obj.d;
  }
}

void oracle_rollout(const OracleModel* m, int precision, const float* pol_w,
                    const float* val_w, int n, const uint32_t* env_ids, double* st,
                    double* pr, int32_t* t_ep, uint32_t* ep, uint64_t t_g0, int T,
                    double* obs, double* act, double* logp, double* value, double* rew,
                    uint8_t* done) {
  if (precision == 1)
    rollout_impl<float>(*m, pol_w, val_w, n, env_ids, st, pr, t_ep, ep, t_g0, T, obs, act,
                        logp, value, rew, done);
  else
    rollout_impl<double>(*m, pol_w, val_w, n, env_ids, st, pr, t_ep, ep, t_g0, T, obs, act,
                         logp, value, rew, done);
}

// Network evaluation on given inputs x[n][in_dim] -> out[n][out_dim].
void oracle_mlp(const float* wts, int in_dim, int hidden, int out_dim, int bf16, int n,
                const double* x, double* out) {
  for (int i = 0; i < n; ++i)
    mlp_forward<double>(wts, in_dim, hidden, out_dim, bf16 != 0, x + (size_t)i * in_dim,
                        out + (size_t)i * out_dim);
}

// Observation and reward terms of one env state (for hand-computed pins).
void oracle_observe(const double* st, const double* pr, double* obs, double* theta_e) {
  int32_t t = 0;
  uint32_t e0 = 0;
  Env<double> e;
  load_env<double>(st, pr, &t, &e0, 1, 0, e);
  observe(e, obs);
  *theta_e = attitude_angle(e);
}

double oracle_reward(const OracleModel* m, const double* st, const double* pr,
                     const double* a_c) {
  int32_t t = 0;
  uint32_t e0 = 0;
  Env<double> e;
  load_env<double>(st, pr, &t, &e0, 1, 0, e);
  return reward(*m, e, a_c);
}

void oracle_allocate(const OracleModel* m, const double* a, double* tau) {
  double a_c[kAct];
  allocate(*m, a, a_c, tau);
}

// Continuous-time nu_dot for one env (state/params SoA with n = 1).
void oracle_nu_dot(const OracleModel* m, const double* st, const double* pr,
                   const double* tau, double* out) {
  int32_t t = 0;
  uint32_t e0 = 0;
  Env<double> e;
  load_env<double>(st, pr, &t, &e0, 1, 0, e);
  nu_dot(*m, e, e.q, e.nu, tau, out);
}

// Physics only: n_steps substeps of size h from the given single-env state
// with constant wrench tau (no reward, no episode logic).  method 0 =
// semi-implicit Euler (the model's integrator), 1 = RK4 brute force.
void oracle_integrate(const OracleModel* m, int method, double* st, const double* pr,
                      const double* tau, double h, int n_steps) {
  int32_t t = 0;
  uint32_t e0 = 0;
  Env<double> e;
  load_env<double>(st, pr, &t, &e0, 1, 0, e);
  for (int s = 0; s < n_steps; ++s) {
    if (method == 0) {
      substep(*m, e, tau, h);
    } else {
      double y[13], k1[13], k2[13], k3[13], k4[13], yt[13];
      for (int k = 0; k < 3; ++k) y[k] = e.p[k];
      for (int k = 0; k < 4; ++k) y[3 + k] = e.q[k];
      for (int k = 0; k < 6; ++k) y[7 + k] = e.nu[k];
      rk4_deriv(*m, e, y, tau, k1);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h / 2 * k1[k];
      rk4_deriv(*m, e, yt, tau, k2);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h / 2 * k2[k];
      rk4_deriv(*m, e, yt, tau, k3);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h * k3[k];
      rk4_deriv(*m, e, yt, tau, k4);
      for (int k = 0; k < 13; ++k) y[k] = y[k] + h / 6 * (k1[k] + 2 * k2[k] + 2 * k3[k] + k4[k]);
      double qn = sqrt(y[3] * y[3] + y[4] * y[4] + y[5] * y[5] + y[6] * y[6]);
      for (int k = 0; k < 3; ++k) e.p[k] = y[k];
      for (int k = 0; k < 4; ++k) e.q[k] = y[3 + k] / qn;
      for (int k = 0; k < 6; ++k) e.nu[k] = y[7 + k];
    }
  }
  store_state(e, 1, 0, st);
}

// ---- the paper's own environment ------------------------------------------
int oracle_paper_model_size() { return (int)sizeof(PaperModel); }

void oracle_paper_reset(const PaperModel* m, int n, const uint32_t* env_ids, double* st,
                        double* pr, int32_t* t_ep, uint32_t* ep) {
  for (int i = 0; i < n; ++i) {
    PaperEnv<double> e;
    std::memset(&e, 0, sizeof(e));
    e.episode = ep[i];
    paper_apply_reset(*m, env_ids[i], e);
    paper_store(e, n, i, st, pr, t_ep, ep);
  }
}

// The paper model's action-replay window objective
// J = sum_t coef[t] r_t + <lam_T, x_T> over its whole state x = (p, q, nu,
// action history: rows 0..60), and the directional derivative along
// (dir_s0 [61][n], dir_act [T][6][n]) in Dual.  The batch is not modified.
void oracle_paper_adjoint_window(const PaperModel* m, int n, const uint32_t* env_ids,
                                 const double* st, const double* pr, const int32_t* t_ep,
                                 const uint32_t* ep, int T, const double* act,
                                 const double* coef, const double* lam_T, const double* dir_s0,
                                 const double* dir_act, double* J, double* dJ) {
  for (int i = 0; i < n; ++i) {
    PaperEnv<Dual> e;
    paper_load<Dual>(st, pr, t_ep, ep, n, i, e);
    for (int k = 0; k < 3; ++k) e.p[k].d = dir_s0[k * n + i];
    for (int k = 0; k < 4; ++k) e.q[k].d = dir_s0[(3 + k) * n + i];
    for (int k = 0; k < 6; ++k) e.nu[k].d = dir_s0[(7 + k) * n + i];
    for (int j = 0; j < kPHist; ++j)
      for (int k = 0; k < 6; ++k) e.hist[j][k].d = dir_s0[(13 + 6 * j + k) * n + i];
    Dual obj = 0.0;
    for (int t = 0; t < T; ++t) {
      Dual a[kPAct];
      for (int k = 0; k < kPAct; ++k) {
        const size_t o = ((size_t)t * kPAct + k) * n + i;
        a[k] = Dual(act[o], dir_act[o]);
      }
      uint8_t d;
      obj += Dual(coef[t]) * paper_control_step(*m, env_ids[i], e, a, &d);
    }
    if (lam_T) {
      for (int k = 0; k < 3; ++k) obj += Dual(lam_T[k * n + i]) * e.p[k];
      for (int k = 0; k < 4; ++k) obj += Dual(lam_T[(3 + k) * n + i]) * e.q[k];
      for (int k = 0; k < 6; ++k) obj += Dual(lam_T[(7 + k) * n + i]) * e.nu[k];
      for (int j = 0; j < kPHist; ++j)
        for (int k = 0; k < 6; ++k) obj += Dual(lam_T[(13 + 6 * j + k) * n + i]) * e.hist[j][k];
    }
    J[i] = obj.v;
    dJ[i] = obj.d;
  }
}

// SHAC's closed-loop window on the paper model: policy 12 -> H -> H -> 12
// (means and log-stds of the 6 wrench commands) acting with the first six
// action normals, the value network at the final observation; J and its
// derivative along the policy-weight direction dpol, in Dual.
void oracle_paper_shac_window(const PaperModel* m, const float* pol_w, const double* dpol,
                              const float* val_w, int n, const uint32_t* env_ids,
                              const double* st, const double* pr, const int32_t* t_ep,
                              const uint32_t* ep, uint64_t t_g0, int T, const double* coef,
                              double coef_V, double* J, double* dJ) {
  for (int i = 0; i < n; ++i) {
    PaperEnv<Dual> e;
    paper_load<Dual>(st, pr, t_ep, ep, n, i, e);
    Dual obj = 0.0;
    for (int t = 0; t < T; ++t) {
      Dual o[kPObs], y[2 * kPAct], a[kPAct];
      paper_observe(e, o);
      mlp_dual(pol_w, dpol, kPObs, m->hidden, 2 * kPAct, o, y);
      uint32_t w[8];
      draw_words(env_ids[i], m->seed, t_g0 + (uint64_t)t, 0u, 2, w);
      float u[8];
      for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
      double eps[8];
      box_muller8(u, eps);
      for (int k = 0; k < kPAct; ++k) {
        Dual ls = y[kPAct + k];
        if (ls < Dual(m->logstd_min)) ls = Dual(m->logstd_min);
        if (ls > Dual(m->logstd_max)) ls = Dual(m->logstd_max);
        a[k] = y[k] + exp(ls) * Dual(eps[k]);
      }
      uint8_t d;
      obj += Dual(coef[t]) * paper_control_step(*m, env_ids[i], e, a, &d);
    }
    if (val_w) {
      Dual o[kPObs], v[1];
      paper_observe(e, o);
      mlp_dual(val_w, nullptr, kPObs, m->hidden, 1, o, v);
      obj += Dual(coef_V) * v[0];
    }
    J[i] = obj.v;
    dJ[i] = obj.d;
  }
}

void oracle_paper_replay(const PaperModel* m, int precision, int n, const uint32_t* env_ids,
                         double* st, double* pr, int32_t* t_ep, uint32_t* ep, int T,
                         const float* act, double* rew, uint8_t* done, double* trace) {
  if (precision == 1)
    paper_replay_impl<float>(*m, n, env_ids, st, pr, t_ep, ep, T, act, rew, done, trace);
  else
    paper_replay_impl<double>(*m, n, env_ids, st, pr, t_ep, ep, T, act, rew, done, trace);
}

void oracle_paper_rollout(const PaperModel* m, int precision, const float* pol_w,
                          const float* val_w, int n, const uint32_t* env_ids, double* st,
                          double* pr, int32_t* t_ep, uint32_t* ep, uint64_t t_g0, int T,
                          double* obs, double* act, double* logp, double* value, double* rew,
                          uint8_t* done) {
  if (precision == 1)
    paper_rollout_impl<float>(*m, pol_w, val_w, n, env_ids, st, pr, t_ep, ep, t_g0, T, obs, act,
                              logp, value, rew, done);
  else
    paper_rollout_impl<double>(*m, pol_w, val_w, n, env_ids, st, pr, t_ep, ep, t_g0, T, obs,
                               act, logp, value, rew, done);
}

// The Gaussian policy's draw for given observations, in double: head =
// network(obs) (bf16 emulation when the model says so), log sigma = the
// clamped head or the fixed vector (A6), eps = the first n_act normals of the
// action-noise stream at global step t_g, a = mu + exp(log sigma) eps and
// log pi(a) = sum(-eps^2/2 - log sigma - log(2 pi)/2), as one step of the
// rollout computes them.  obs[n][obs_dim] row-major; act[n][n_act], logp[n]
// and, if mu is not NULL, the mean mu[n][n_act].
void oracle_policy_act(const OracleModel* m, const float* pol_w, int n,
                       const uint32_t* env_ids, uint64_t t_g, const double* obs, double* act,
                       double* logp, double* mu_out) {
  const double half_log_2pi = 0.91893853320467274178032973640562;
  for (int i = 0; i < n; ++i) {
    double mu[kAct], logstd[kAct];
    policy_head<double>(*m, pol_w, obs + (size_t)i * kObs, mu, logstd);
    uint32_t w[8];
    draw_words(env_ids[i], m->seed, t_g, 0u, 2, w);
    float u[8];
    for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
    double eps[8];
    box_muller8(u, eps);
    double lp = 0;
    for (int k = 0; k < kAct; ++k) {
      act[(size_t)i * kAct + k] = mu[k] + std::exp(logstd[k]) * eps[k];
      lp += -0.5 * eps[k] * eps[k] - logstd[k] - half_log_2pi;
      if (mu_out) mu_out[(size_t)i * kAct + k] = mu[k];
    }
    logp[i] = lp;
  }
}

void oracle_paper_policy_act(const PaperModel* m, const float* pol_w, int n,
                             const uint32_t* env_ids, uint64_t t_g, const double* obs,
                             double* act, double* logp, double* mu_out) {
  const double half_log_2pi = 0.91893853320467274178032973640562;
  for (int i = 0; i < n; ++i) {
    double out[12];
    mlp_forward<double>(pol_w, kPObs, m->hidden, m->policy_out, m->mlp_bf16 != 0,
                        obs + (size_t)i * kPObs, out);
    uint32_t w[8];
    draw_words(env_ids[i], m->seed, t_g, 0u, 2, w);
    float u[8];
    for (int k = 0; k < 8; ++k) u[k] = word_to_uniform(w[k]);
    double eps[8];
    box_muller8(u, eps);
    double lp = 0;
    for (int k = 0; k < kPAct; ++k) {
      double ls = (double)m->logstd_fixed[k];
      if (m->policy_out == 12) {
        ls = out[kPAct + k];
        ls = ls < (double)m->logstd_min ? (double)m->logstd_min : ls;
        ls = ls > (double)m->logstd_max ? (double)m->logstd_max : ls;
      }
      act[(size_t)i * kPAct + k] = out[k] + std::exp(ls) * eps[k];
      lp += -0.5 * eps[k] * eps[k] - ls - half_log_2pi;
      if (mu_out) mu_out[(size_t)i * kPAct + k] = out[k];
    }
    logp[i] = lp;
  }
}

// Observation of one env (SoA with n = 1).
void oracle_paper_observe(const double* st, const double* pr, double* obs) {
  int32_t t = 0;
  uint32_t e0 = 0;
  PaperEnv<double> e;
  paper_load<double>(st, pr, &t, &e0, 1, 0, e);
  paper_observe(e, obs);
}

// Reward of one env's (post-step) state with clipped action a_c and its history.
double oracle_paper_reward(const PaperModel* m, const double* st, const double* pr,
                           const double* a_c) {
  int32_t t = 0;
  uint32_t e0 = 0;
  PaperEnv<double> e;
  paper_load<double>(st, pr, &t, &e0, 1, 0, e);
  return paper_reward(*m, e, a_c);
}

void oracle_paper_wrench(const PaperModel* m, const double* a, double* a_c, double* tau) {
  paper_wrench(*m, a, a_c, tau);
}

void oracle_paper_box(const PaperModel* m, double* b) { paper_box(*m, b); }

void oracle_paper_nu_dot(const PaperModel* m, const double* st, const double* pr,
                         const double* tau, double* out) {
  int32_t t = 0;
  uint32_t e0 = 0;
  PaperEnv<double> e;
  paper_load<double>(st, pr, &t, &e0, 1, 0, e);
  paper_nu_dot(*m, e, e.q, e.nu, tau, out);
}

// Physics only, constant wrench: method 0 = the model's integrator, 1 = RK4.
void oracle_paper_integrate(const PaperModel* m, int method, double* st, const double* pr,
                            const double* tau, double h, int n_steps) {
  int32_t t = 0;
  uint32_t e0 = 0;
  PaperEnv<double> e;
  paper_load<double>(st, pr, &t, &e0, 1, 0, e);
  for (int s = 0; s < n_steps; ++s) {
    if (method == 0) {
      paper_substep(*m, e, tau, h);
    } else {
      double y[13], k1[13], k2[13], k3[13], k4[13], yt[13];
      for (int k = 0; k < 3; ++k) y[k] = e.p[k];
      for (int k = 0; k < 4; ++k) y[3 + k] = e.q[k];
      for (int k = 0; k < 6; ++k) y[7 + k] = e.nu[k];
      paper_rk4_deriv(*m, e, y, tau, k1);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h / 2 * k1[k];
      paper_rk4_deriv(*m, e, yt, tau, k2);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h / 2 * k2[k];
      paper_rk4_deriv(*m, e, yt, tau, k3);
      for (int k = 0; k < 13; ++k) yt[k] = y[k] + h * k3[k];
      paper_rk4_deriv(*m, e, yt, tau, k4);
      for (int k = 0; k < 13; ++k) y[k] = y[k] + h / 6 * (k1[k] + 2 * k2[k] + 2 * k3[k] + k4[k]);
      double qn = sqrt(y[3] * y[3] + y[4] * y[4] + y[5] * y[5] + y[6] * y[6]);
      for (int k = 0; k < 3; ++k) e.p[k] = y[k];
      for (int k = 0; k < 4; ++k) e.q[k] = y[3 + k] / qn;
      for (int k = 0; k < 6; ++k) e.nu[k] = y[7 + k];
    }
  }
  paper_store_state(e, 1, 0, st);
}

}  // extern "C"
