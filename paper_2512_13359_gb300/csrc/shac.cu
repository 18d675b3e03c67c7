// shac.cu -- SHAC's actor gradient over a window in closed loop (paper §III-A:
// short-horizon actor-critic; Xu et al. 2022): the policy acts through the
// differentiable step for T steps, and back-propagation through the
// dynamics, the policy network and the observation gives dJ/dtheta of
//   J = sum_i [ sum_t coef_t r_t,i + coef_V V(o_T,i) ]
// (theta: the policy weights; V: the terminal critic; actions reparameterised
// as a = mu(o) + exp(clamp(ls(o))) eps with the rollout's action noise eps).
//
// Per step the per-env work (observation, action, physics and their VJPs)
// runs in the k_shac_* kernels of k_adjoint.cu; the policy network's dense
// products run in the library's GEMM (k_gemm.cu: tcgen05 with tf32 operands,
// or fp32 on the CUDA cores) on the augmented layout of the PPO learner (a
// constant-1 input column carries each bias).  Forward: for each
// step, observation -> policy GEMMs (activations kept for every step) ->
// action and physics (the env advances).  Backward, t = T-1 .. 0: physics
// VJP of step t (the state adjoint lam and the head gradient), the policy's
// backward (weight gradients accumulated over steps, input gradient), then
// the observation VJP into lam.  The terminal critic seeds lam with
// coef_V dV(o(x_T))/dx_T through the value network's input gradient.
#include <algorithm>
#include <cstdio>

#include "auv_gemm.h"
#include "auv_kernels.h"
#include "auvenv.h"
#include "paper_device.cuh"

namespace auv {
namespace shac {

namespace {

int round8(int x) { return (x + 7) & ~7; }

// C = op(A) op(B) (+ beta C) in column-major terms (ta / tb: the operand is
// transposed), fp32 operands and result: the row-major product
// C'[n][m] = sum_k opB(k, n) opA(m, k) on the library's GEMM.
struct Gemm {
  bool tf32;
  float* ws;
  size_t ws_bytes;
  Status* st;
  cudaStream_t s;
  cudaError_t operator()(bool ta, bool tb, int m, int n, int k, const float* A, int lda,
                         const float* B, int ldb, float* C, int ldc, float beta = 0.0f) const {
    const gemm::Operand a = {B, ldb, tb}, b = {A, lda, !ta};
    return gemm::launch(tf32 ? gemm::kTf32 : gemm::kFp32, n, m, k, a, b, C, ldc, false, beta, ws,
                        ws_bytes, st, s);
  }
};

constexpr int kLdy = 16;   // policy head row (2 x 8, or 2 x 6 padded)
constexpr int kLdv = 8;    // value head row

}  // namespace

Layout layout(int n, int T, int H, bool paper) {
  Layout L;
  L.n = n;
  L.T = T;
  L.H = H;
  L.D = paper ? paper::kObs : kObs;
  L.out = 2 * (paper ? paper::kAct : kAct);
  L.S = paper ? paper::kStateF : 13;
  L.Dp = round8(L.D + 1);
  L.Hp = round8(H + 1);
  L.n_aug_p = ppo::aug_count(L.D, L.Dp, H, L.Hp, L.out);
  L.n_aug_v = ppo::aug_count(L.D, L.Dp, H, L.Hp, 1);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return o;
  };
  const size_t N = (size_t)n;
  L.o_X = take((T + 1) * N * L.Dp * 4);
  L.o_H1 = take(T * N * L.Hp * 4);
  L.o_H2 = take(T * N * L.Hp * 4);
  L.o_Y = take(T * N * kLdy * 4);
  L.o_G = take(N * H * 4);
  L.o_GX = take(N * L.Dp * 4);
  L.o_gY = take(N * kLdy * 4);
  L.o_lam = take((size_t)L.S * N * 4);
  L.o_done = take(T * N);
  L.o_rew = take(T * N * 4);
  L.o_VH1 = take(N * L.Hp * 4);
  L.o_VH2 = take(N * L.Hp * 4);
  L.o_V = take(N * kLdv * 4);
  L.o_gYv = take(N * kLdv * 4);
  L.o_wp = take(L.n_aug_p * 4);
  L.o_wv = take(L.n_aug_v * 4);
  L.o_gp = take(L.n_aug_p * 4);
  L.o_sc = take(adjoint_scratch_floats(n, T) * 4);
  // the GEMM workspace of the largest product (policy and value networks)
  size_t gws = 0;
  for (int o : {L.out, 1}) {
    const int shapes[9][3] = {{n, H, L.Dp}, {n, H, L.Hp}, {n, o, L.Hp},   {o, L.Hp, n},    {n, H, o},
                              {H, L.Hp, n}, {n, H, H},    {H, L.Dp, n}, {n, L.Dp, H}};
    for (const auto& sh : shapes) gws = std::max(gws, gemm::workspace_bytes(sh[0], sh[1], sh[2]));
  }
  L.o_gws = take(gws);
  L.gws_bytes = gws;
  L.bytes = off;
  return L;
}

cudaError_t init(const Layout& L, char* base, cudaStream_t s) {
  cudaError_t e = cudaMemsetAsync(base, 0, L.bytes, s);
  float* h1 = reinterpret_cast<float*>(base + L.o_H1);
  float* h2 = reinterpret_cast<float*>(base + L.o_H2);
  const int rows = L.T * L.n;
  if (e == cudaSuccess) e = ppo::launch_fill_ones(false, h1, L.Hp, L.H, rows, s);
  if (e == cudaSuccess) e = ppo::launch_fill_ones(false, h2, L.Hp, L.H, rows, s);
  if (e == cudaSuccess)
    e = ppo::launch_fill_ones(false, base + L.o_VH1, L.Hp, L.H, L.n, s);
  if (e == cudaSuccess)
    e = ppo::launch_fill_ones(false, base + L.o_VH2, L.Hp, L.H, L.n, s);
  return e;
}

int run_window(const Model& M, const Buffers& B, Status* st, const Layout& L,
               char* base, uint64_t t_g0, const float* policy, const float* value,
               const float* coef, float coef_V, bool tf32, float* grad, float* J,
               float* obs_out, float* rew_out, uint8_t* done_out, cudaStream_t s, char* err) {
  const int n = L.n, T = L.T, H = L.H, Dp = L.Dp, Hp = L.Hp;
  const size_t N = (size_t)n;
  auto F = [&](size_t o) { return reinterpret_cast<float*>(base + o); };
  float *X = F(L.o_X), *H1 = F(L.o_H1), *H2 = F(L.o_H2), *Y = F(L.o_Y), *G = F(L.o_G),
        *GX = F(L.o_GX), *gY = F(L.o_gY), *lam = F(L.o_lam), *rew = F(L.o_rew),
        *VH1 = F(L.o_VH1), *VH2 = F(L.o_VH2), *V = F(L.o_V), *gYv = F(L.o_gYv),
        *wp = F(L.o_wp), *wv = F(L.o_wv), *gp = F(L.o_gp), *sc = F(L.o_sc);
  uint8_t* done = reinterpret_cast<uint8_t*>(base + L.o_done);
  auto Xs = [&](int t) { return X + (size_t)t * N * Dp; };
  auto H1s = [&](int t) { return H1 + (size_t)t * N * Hp; };
  auto H2s = [&](int t) { return H2 + (size_t)t * N * Hp; };
  auto Ys = [&](int t) { return Y + (size_t)t * N * kLdy; };
  auto SCs = [&](int t) { return sc + (size_t)t * adjoint_step_floats(n); };
  const float *w1 = wp, *w2 = wp + (size_t)H * Dp, *w3 = w2 + (size_t)H * Hp;
  float *g1 = gp, *g2 = gp + (size_t)H * Dp, *g3 = g2 + (size_t)H * Hp;
  const float *v1 = wv, *v2 = wv + (size_t)H * Dp, *v3 = v2 + (size_t)H * Hp;

  const Gemm gemm{tf32, F(L.o_gws), L.gws_bytes, st, s};
  cudaError_t e = cudaSuccess;
  auto cfail = [&](cudaError_t x, const char* what) {
    snprintf(err, 256, "%s: %s", what, cudaGetErrorString(x));
    return AUV_ERR_CUDA;
  };
  const bool T_ = true, N_ = false;

  // weights into the augmented layout; gradient accumulator to zero
  const int D = L.D, out = L.out;
  if ((e = ppo::launch_convert(const_cast<float*>(policy), wp, D, Dp, H, Hp, out, true, s)))
    return cfail(e, "policy weights");
  if (value &&
      (e = ppo::launch_convert(const_cast<float*>(value), wv, D, Dp, H, Hp, 1, true, s)))
    return cfail(e, "value weights");
  if ((e = cudaMemsetAsync(gp, 0, L.n_aug_p * 4, s))) return cfail(e, "clear gradient");

  // ---- forward ----
  for (int t = 0; t < T; ++t) {
    if ((e = launch_obs(M, B, SCs(t), Xs(t), Dp, obs_out, t, s))) return cfail(e, "observation");
    if ((e = gemm(T_, N_, H, n, Dp, w1, Dp, Xs(t), Dp, H1s(t), Hp))) return cfail(e, "policy 1");
    if ((e = ppo::launch_tanh_fwd(false, H1s(t), Hp, n, H, s))) return cfail(e, "tanh");
    if ((e = gemm(T_, N_, H, n, Hp, w2, Hp, H1s(t), Hp, H2s(t), Hp))) return cfail(e, "policy 2");
    if ((e = ppo::launch_tanh_fwd(false, H2s(t), Hp, n, H, s))) return cfail(e, "tanh");
    if ((e = gemm(T_, N_, out, n, Hp, w3, Hp, H2s(t), Hp, Ys(t), kLdy)))
      return cfail(e, "policy 3");
    if ((e = launch_step(M, B, Ys(t), kLdy, t_g0 + (uint64_t)t, rew + (size_t)t * N,
                         done + (size_t)t * N, st, s)))
      return cfail(e, "step");
  }
  if ((e = cudaMemsetAsync(lam, 0, (size_t)L.S * N * 4, s))) return cfail(e, "clear adjoint");
  // ---- terminal critic: lam = coef_V dV(o(x_T))/dx_T ----
  if (value) {
    if ((e = launch_obs(M, B, nullptr, Xs(T), Dp, nullptr, 0, s))) return cfail(e, "observation");
    if ((e = gemm(T_, N_, H, n, Dp, v1, Dp, Xs(T), Dp, VH1, Hp))) return cfail(e, "value 1");
    if ((e = ppo::launch_tanh_fwd(false, VH1, Hp, n, H, s))) return cfail(e, "tanh");
    if ((e = gemm(T_, N_, H, n, Hp, v2, Hp, VH1, Hp, VH2, Hp))) return cfail(e, "value 2");
    if ((e = ppo::launch_tanh_fwd(false, VH2, Hp, n, H, s))) return cfail(e, "tanh");
    if ((e = gemm(T_, N_, 1, n, Hp, v3, Hp, VH2, Hp, V, kLdv))) return cfail(e, "value 3");
    if ((e = launch_fill_col(n, gYv, kLdv, coef_V, s))) return cfail(e, "critic seed");
    if ((e = gemm(N_, N_, H, n, 1, v3, Hp, gYv, kLdv, G, H))) return cfail(e, "value dH2");
    if ((e = ppo::launch_tanh_bwd(false, G, H, VH2, Hp, n, H, s))) return cfail(e, "tanh'");
    if ((e = gemm(N_, N_, H, n, H, v2, Hp, G, H, VH2, Hp))) return cfail(e, "value dH1");
    if ((e = ppo::launch_tanh_bwd(false, VH2, Hp, VH1, Hp, n, H, s))) return cfail(e, "tanh'");
    if ((e = gemm(N_, N_, Dp, n, H, v1, Dp, VH2, Hp, GX, Dp))) return cfail(e, "value dX");
    if ((e = launch_obs_vjp(M, B, nullptr, GX, Dp, lam, s))) return cfail(e, "observation VJP");
  }
  if (J && (e = launch_objective(n, T, rew, coef, value ? V : nullptr, kLdv, coef_V, J, s)))
    return cfail(e, "objective");
  // ---- backward through the window ----
  for (int t = T - 1; t >= 0; --t) {
    if ((e = launch_bwd(M, SCs(t), Ys(t), kLdy, done + (size_t)t * N, t_g0 + (uint64_t)t,
                        coef + t, lam, gY, s)))
      return cfail(e, "step VJP");
    if ((e = gemm(N_, T_, Hp, out, n, H2s(t), Hp, gY, kLdy, g3, Hp, 1.0f)))
      return cfail(e, "dW3");
    if ((e = gemm(N_, N_, H, n, out, w3, Hp, gY, kLdy, G, H))) return cfail(e, "dH2");
    if ((e = ppo::launch_tanh_bwd(false, G, H, H2s(t), Hp, n, H, s))) return cfail(e, "tanh'");
    if ((e = gemm(N_, T_, Hp, H, n, H1s(t), Hp, G, H, g2, Hp, 1.0f))) return cfail(e, "dW2");
    if ((e = gemm(N_, N_, H, n, H, w2, Hp, G, H, H2s(t), Hp))) return cfail(e, "dH1");
    if ((e = ppo::launch_tanh_bwd(false, H2s(t), Hp, H1s(t), Hp, n, H, s)))
      return cfail(e, "tanh'");
    if ((e = gemm(N_, T_, Dp, H, n, Xs(t), Dp, H2s(t), Hp, g1, Dp, 1.0f))) return cfail(e, "dW1");
    if ((e = gemm(N_, N_, Dp, n, H, w1, Dp, H2s(t), Hp, GX, Dp))) return cfail(e, "dX");
    if ((e = launch_obs_vjp(M, B, SCs(t), GX, Dp, lam, s))) return cfail(e, "observation VJP");
  }
  if ((e = ppo::launch_convert(grad, gp, D, Dp, H, Hp, out, false, s)))
    return cfail(e, "gradient layout");
  if (rew_out && (e = cudaMemcpyAsync(rew_out, rew, T * N * 4, cudaMemcpyDefault, s)))
    return cfail(e, "copy rewards");
  if (done_out && (e = cudaMemcpyAsync(done_out, done, T * N, cudaMemcpyDefault, s)))
    return cfail(e, "copy dones");
  return AUV_OK;
}

}  // namespace shac
}  // namespace auv
