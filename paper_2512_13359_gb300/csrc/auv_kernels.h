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

// Reverse-mode adjoint of the Fossen control step over an action window
// (k_adjoint.cu).  scratch: adjoint_scratch_floats(n, T) floats.  T <= 64,
// M.substeps <= 8.
size_t adjoint_scratch_floats(int n, int T);
size_t adjoint_step_floats(int n);   // one Fossen step's slice of the scratch
cudaError_t launch_adjoint(const Model& M, const Buffers& B, const float* act, int T,
                           const float* coef, const float* lam_T, float* g_act, float* lam_0,
                           float* rew, uint8_t* done, float* scratch, Status* st,
                           cudaStream_t s);

// SHAC in closed loop (k_adjoint.cu kernels, shac.cu orchestration).
namespace shac {
struct Layout {
  int n, T, H, Dp, Hp;
  int D, out, S;     // network input, policy head width, adjoint rows (model)
  size_t n_aug_p, n_aug_v;
  size_t o_X, o_H1, o_H2, o_Y, o_G, o_GX, o_gY, o_lam, o_done, o_rew, o_VH1, o_VH2, o_V, o_gYv,
      o_wp, o_wv, o_gp, o_sc, o_gws, gws_bytes, bytes;
};
// paper: the paper model (input 12, head 12, 61 adjoint rows), else Fossen
// (18, 16, 13).
Layout layout(int n, int T, int H, bool paper);
cudaError_t init(const Layout& L, char* base, cudaStream_t s);
// Returns AUV_OK or an AUV_ERR_* code with err set.
int run_window(const Model& M, const Buffers& B, Status* st, const Layout& L,
               char* base, uint64_t t_g0, const float* policy, const float* value,
               const float* coef, float coef_V, bool tf32, float* grad, float* J,
               float* obs_out, float* rew_out, uint8_t* done_out, cudaStream_t s, char* err);
// obs_fm: optional [T][18][N] output of step t's observation.
cudaError_t launch_obs(const Model& M, const Buffers& B, float* sc, float* X, int ldx,
                       float* obs_fm, int t, cudaStream_t s);
cudaError_t launch_step(const Model& M, const Buffers& B, const float* Y, int ldy, uint64_t t_g,
                        float* rew, uint8_t* done, Status* st, cudaStream_t s);
cudaError_t launch_bwd(const Model& M, const float* sc, const float* Y, int ldy,
                       const uint8_t* done, uint64_t t_g, const float* coef, float* lam,
                       float* gY, cudaStream_t s);
cudaError_t launch_obs_vjp(const Model& M, const Buffers& B, const float* sc, const float* gX,
                           int ldx, float* lam, cudaStream_t s);
cudaError_t launch_objective(int n, int T, const float* rew, const float* coef, const float* V,
                             int ldv, float coef_V, float* J, cudaStream_t s);
cudaError_t launch_fill_col(int n, float* buf, int ld, float v, cudaStream_t s);
}  // namespace shac

// Inverse thruster allocation (rbuf.cu): commands = clip(pinv u-map, -1, 1).
struct InvAlloc {
  float pinv[48];   // [8][6]: pseudo-inverse of alloc * thrust_max
};
bool pinv_6x8(const float* alloc_t, float* out);
cudaError_t launch_inverse_alloc(int n, const InvAlloc& ia, const float* wrench, float* cmd,
                                 cudaStream_t s);

// PPO learner pieces (k_ppo.cu)
cudaError_t launch_gae(int n, int T, const float* rew, const uint8_t* done, const float* value,
                       const float* last_value, float gamma, float lam, float* adv, float* ret,
                       cudaStream_t s);

namespace ppo {

// Shapes of one learner.  Each network is held "augmented": every layer's
// input row carries a constant 1 after its features (then zeros up to a
// multiple of 4 floats), and the layer's bias is the weight column that
// meets it, so that a GEMM adds the bias and the weight-gradient GEMM yields
// its gradient.  W1a [H][Dp], W2a [H][Hp], W3a [out][Hp].
struct Dims {
  int D, Dp;     // observation width and its padded, augmented row (>= D + 1)
  int A;         // action width; policy head 2A
  int H, Hp;     // hidden width and its augmented row (>= H + 1)
  int Ha;        // row length of the activation arrays H1, H2 (>= Hp; bf16: a
                 // multiple of 16, so that rows start on 32-byte boundaries)
  int B;         // minibatch
  int ld_pol;    // row length of the policy head arrays Y, dL/dY (>= 2A)
  int ld_val;    // row length of the value head arrays (>= 1)
  int bf16;      // activations and head gradients stored as bf16
  int value_only;  // critic regression: the policy is not run
};

struct PermKey {        // Feistel permutation of [0, m) for one epoch
  uint32_t m, mask;
  int h;                // half width in bits
  uint32_t k0, k1, e0, e1;
};

struct LossHp {
  float clip_eps, vf_coef, ent_coef, logstd_min, logstd_max;
  int norm_adv;
};

struct AdamHp {
  float lr, b1, b2, eps;
  float max_norm;
};

// Per-step variables of an update, in device memory so that one captured
// step (a CUDA graph) can be replayed: step s of the update gathers
// minibatch s mod n_mb of epoch epoch0 + s / n_mb, and Adam takes its step
// t + 1 (bias corrections 1 - b^(t+1)); launch_step_advance then moves to
// the next step.
struct StepCtl {
  unsigned long long epoch0;
  unsigned long long t;
  unsigned int n_mb;
  unsigned int step;
};

struct Sample {                    // gathered minibatch, sample-major
  float* act;                      // [B][A]
  float* logp;                     // [B]
  float* adv;                      // [B]
  float* ret;                      // [B]
  double* adv_part;                // [ceil(B/256)][2]: sums of adv and adv^2
};

constexpr int kNormBlocks = 256;   // blocks of the gradient-norm reduction

size_t aug_count(int in, int in_p, int H, int Hp, int out);
// X [B][Dp]: the gathered observations with the constant 1 at column D,
// fp32 or bf16 (Dims::bf16), as are the activation arguments below.
// k: the permutation of the batch's rows (its epoch words are taken from ctl).
cudaError_t launch_gather(const Dims& d, const PermKey& k, const StepCtl* ctl, const float* obs,
                          const float* act, const float* logp, const float* adv,
                          const float* ret, uint32_t N, const Sample& out, void* X,
                          cudaStream_t s);
cudaError_t launch_step_advance(StepCtl* ctl, cudaStream_t s);
cudaError_t launch_tanh_fwd(bool bf16, void* h, int ld, int B, int H, cudaStream_t s);
// Sample-major copy of a batch for the gather: rows of sample_row_floats(D, A)
// floats (obs, act, logp, adv, ret, zero padding), row r = t N + i; act,
// logp and adv may be NULL (value-only).  D + A + 3 <= 80.
int sample_row_floats(int D, int A);
cudaError_t launch_transpose_batch(int D, int A, uint32_t T, uint32_t N, const float* obs,
                                   const float* act, const float* logp, const float* adv,
                                   const float* ret, float* dst, cudaStream_t s);
cudaError_t launch_gather_sm(const Dims& d, const PermKey& k, const StepCtl* ctl,
                             const float* rows, const Sample& out, void* X, cudaStream_t s);
cudaError_t launch_tanh_bwd(bool bf16, void* g, int ldg, const void* h, int ldh, int B, int H,
                            cudaStream_t s);
// y [B][ld_pol], v [B][ld_val] fp32 head outputs; g_y, g_v the same shapes.
cudaError_t launch_head(const Dims& d, const LossHp& hp, const float* y, const float* v,
                        const Sample& smp, void* g_y, void* g_v, float* part, cudaStream_t s);
cudaError_t launch_stats(const Dims& d, const LossHp& hp, const float* part, float* mb,
                         float* acc, cudaStream_t s);
// wb (bf16 copy of w, may be NULL) is rewritten with the new weights.
// part: kNormBlocks + 3 floats (norm partials, then the step's scalars).
cudaError_t launch_adam(float* w, const float* g, float* m, float* v, size_t n, float* part,
                        const AdamHp& hp, const StepCtl* ctl, float* mb, float* acc, void* wb,
                        cudaStream_t s);
cudaError_t launch_to_bf16(const float* w, void* wb, size_t n, cudaStream_t s);
cudaError_t launch_finish(const float* acc, float* out, cudaStream_t s);
// flat [W1|b1|W2|b2|W3|b3] <-> augmented [W1a|W2a|W3a] of one network
cudaError_t launch_convert(float* flat, float* aug, int in, int in_p, int H, int Hp, int out,
                           bool to_aug, cudaStream_t s);
// the same for the policy and the value network in one launch
cudaError_t launch_convert_pair(float* flat_pol, float* aug_pol, int out_pol, float* flat_val,
                                float* aug_val, int out_val, int in, int in_p, int H, int Hp,
                                bool to_aug, cudaStream_t s);
cudaError_t launch_fill_ones(bool bf16, void* buf, int ld, int col, int rows, cudaStream_t s);

}  // namespace ppo

}  // namespace auv
