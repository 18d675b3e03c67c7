// ppo_api.cu -- the PPO learner's extern "C" entry points (include/auvenv.h):
// validation, the learner's device memory, and the sequence of one gradient
// step: gather -> forward GEMMs + tanh -> loss head -> backward GEMMs + tanh'
// -> (gradient norm, Adam).  The dense products run in the library's GEMM
// (k_gemm.cu) and, in bf16 mode, the forward and backward-data passes on the
// tensor-core engine (k_bf16.cu); every other step runs in the kernels of
// k_ppo.cu.  Precision modes:
//   fp32  fp32 activations, fp32 GEMMs on the CUDA cores;
//   tf32  fp32 activations, tensor-core GEMMs with tf32 operands;
//   bf16  bf16 activations, backward signals and weight copy (the GEMM
//         operands), tensor-core GEMMs with fp32 sums; the heads' outputs
//         and the weight gradients stay fp32, as do the master weights.
//
// Memory layout (one cudaMalloc): master weights, gradient and Adam moments
// as augmented vectors [policy | value] (auv_kernels.h, ppo::Dims), the bf16
// weight copy, a flat staging vector, the gathered minibatch, and per
// network the activations H1, H2 [B][Hp] (constant 1 at column H), the
// backward buffer G [B][H] and the head output Y [B][ld].  Everything a step
// touches is resident.  ppo_update adds one separate allocation: a
// sample-major copy of its batch (rows of round8(D + A + 3) floats), made
// once per call, from which every step gathers its minibatch; it grows when a
// larger batch arrives and lives until ppo_destroy.

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>

#include <climits>

#include "auv_bf16.h"
#include "auv_device.cuh"
#include "auv_gemm.h"
#include "auv_kernels.h"
#include "auvenv.h"

namespace ppo = auv::ppo;
using auv::Status;

struct auv_ppo {
  auv_ppo_config cfg;
  int device;
  ppo::Dims d;
  int out[2];                 // head widths: 2A (policy), 1 (value)
  size_t n_flat[2], n_aug[2], n_aug_all;
  char* mem;
  bool bf16;
  size_t esz;                 // its size in bytes
  float *w, *g, *m, *v;       // augmented [policy | value]
  void* wb;                   // bf16 copy of w (bf16 mode)
  float* flat;                // staging, flat [policy | value]
  ppo::Sample smp;
  void* X;                    // [B][Dp]
  void *h1[2], *h2[2], *gb[2];
  float* y[2];                // head outputs [B][ld_pol], [B][ld_val]
  void *g_y, *g_v;            // dL/d(head), same shapes
  float *head_part, *norm_part;
  float *mb, *acc;            // statistics records (AUV_PPO_STATS floats)
  ppo::StepCtl* ctl;          // device: per-step variables
  float* gws;                 // GEMM workspace: split-K partials, tf32 transposes
  size_t gws_bytes;
  // bf16 forward and backward-data on the tensor-core engine: packed images
  // of both networks (forward, and transposed for the backward), rebuilt
  // from w every step, a flat staging copy and a status block
  bool eng = false;
  void *img_p = nullptr, *img_v = nullptr, *img_bp = nullptr, *img_bv = nullptr;
  float* flat_eng = nullptr;
  Status* st = nullptr;
  // sample-major copy of the batch of the current ppo_update (use_sm while
  // that update's steps are enqueued); the step graph records which copy
  float* sm_buf = nullptr;
  size_t sm_rows = 0;
  bool use_sm = false;
  const float* graph_sm = nullptr;
  uint64_t t, epoch;
  // One gradient step captured as a CUDA graph for ppo_update, replayed on a
  // private stream; valid for the batch it was captured with.
  cudaStream_t gstream = nullptr;
  cudaEvent_t ev_in = nullptr, ev_out = nullptr;
  cudaGraphExec_t step_graph = nullptr;
  auv_ppo_batch graph_batch;
  bool graph_failed = false;
  char err[256];
};

namespace {

thread_local char g_err[256] = "";

int fail(auv_ppo* p, int code, const char* fmt, ...) {
  char* dst = p ? p->err : g_err;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(dst, 256, fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(auv_ppo* p, cudaError_t e, const char* what) {
  return fail(p, AUV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}


int round8(int x) { return (x + 7) & ~7; }

bool is_device(const void* q) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, q) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged;
}

int check_dev(auv_ppo* p, const void* q, const char* name) {
  if (!q) return fail(p, AUV_ERR_INVALID, "%s is NULL", name);
  if (reinterpret_cast<uintptr_t>(q) % 4) return fail(p, AUV_ERR_SIZE, "%s not 4-byte aligned", name);
  if (!is_device(q)) return fail(p, AUV_ERR_SIZE, "%s is not device memory", name);
  return AUV_OK;
}

int check_device(auv_ppo* p) {
  int cur = -1;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return cuda_fail(p, e, "cudaGetDevice");
  if (cur != p->device)
    return fail(p, AUV_ERR_INVALID, "device %d is current but the learner lives on device %d",
                cur, p->device);
  return AUV_OK;
}

int validate(const auv_ppo_config* c) {
  if (!c) return fail(nullptr, AUV_ERR_INVALID, "cfg is NULL");
  if (c->struct_size != sizeof(auv_ppo_config))
    return fail(nullptr, AUV_ERR_INVALID, "cfg->struct_size %u != sizeof(auv_ppo_config) %zu",
                c->struct_size, sizeof(auv_ppo_config));
  if (c->obs_dim < 1 || c->obs_dim > 64) return fail(nullptr, AUV_ERR_INVALID, "obs_dim outside [1, 64]");
  if (c->act_dim < 1 || c->act_dim > 8) return fail(nullptr, AUV_ERR_INVALID, "act_dim outside [1, 8]");
  if (c->hidden < 8 || c->hidden > 1024 || c->hidden % 8)
    return fail(nullptr, AUV_ERR_INVALID, "hidden must be a multiple of 8 in [8, 1024]");
  if (c->minibatch < 2 || c->minibatch > (1u << 22))
    return fail(nullptr, AUV_ERR_INVALID, "minibatch outside [2, 2^22]");
  if (c->precision > AUV_PPO_BF16) return fail(nullptr, AUV_ERR_INVALID, "unknown precision %u", c->precision);
  if (c->norm_adv > 1) return fail(nullptr, AUV_ERR_INVALID, "norm_adv must be 0 or 1");
  if (c->flags & ~(AUV_PPO_VALUE_ONLY | AUV_PPO_GEMM_PATH))
    return fail(nullptr, AUV_ERR_INVALID, "unknown flags %#x", c->flags);
  if (!(std::isfinite(c->clip_eps) && c->clip_eps > 0.0f))
    return fail(nullptr, AUV_ERR_INVALID, "clip_eps must be finite and > 0");
  if (!std::isfinite(c->vf_coef) || !std::isfinite(c->ent_coef) || std::isnan(c->max_grad_norm) ||
      std::isinf(c->max_grad_norm))
    return fail(nullptr, AUV_ERR_INVALID, "loss coefficients and max_grad_norm must be finite");
  if (!(std::isfinite(c->lr) && c->lr >= 0.0f)) return fail(nullptr, AUV_ERR_INVALID, "lr must be finite and >= 0");
  if (!(c->adam_beta1 >= 0.0f && c->adam_beta1 < 1.0f && c->adam_beta2 >= 0.0f && c->adam_beta2 < 1.0f))
    return fail(nullptr, AUV_ERR_INVALID, "Adam betas must lie in [0, 1)");
  if (!(std::isfinite(c->adam_eps) && c->adam_eps > 0.0f))
    return fail(nullptr, AUV_ERR_INVALID, "adam_eps must be finite and > 0");
  if (!(std::isfinite(c->logstd_min) && std::isfinite(c->logstd_max) && c->logstd_min <= c->logstd_max))
    return fail(nullptr, AUV_ERR_INVALID, "logstd clamp invalid");
  return AUV_OK;
}

int check_batch(auv_ppo* p, const auv_ppo_batch* b) {
  if (!b) return fail(p, AUV_ERR_INVALID, "batch is NULL");
  if (b->T < 1 || b->N < 1) return fail(p, AUV_ERR_INVALID, "batch T and N must be >= 1");
  if ((uint64_t)b->T * b->N > (1ull << 31)) return fail(p, AUV_ERR_SIZE, "T * N exceeds 2^31");
  int rc;
  if ((rc = check_dev(p, b->obs, "batch.obs")) || (rc = check_dev(p, b->ret, "batch.ret")))
    return rc;
  if (p->d.value_only) return AUV_OK;     // act, logp, adv are not read
  if ((rc = check_dev(p, b->act, "batch.act")) || (rc = check_dev(p, b->logp, "batch.logp")) ||
      (rc = check_dev(p, b->adv, "batch.adv")))
    return rc;
  return AUV_OK;
}

ppo::PermKey perm_key(const auv_ppo* p, uint32_t m, uint64_t epoch) {
  ppo::PermKey k;
  int bits = 2;
  while ((1ull << bits) < m) bits += 2;
  k.m = m;
  k.h = bits / 2;
  k.mask = k.h >= 32 ? 0xFFFFFFFFu : ((1u << k.h) - 1u);
  k.k0 = (uint32_t)p->cfg.seed;
  k.k1 = (uint32_t)(p->cfg.seed >> 32);
  k.e0 = (uint32_t)epoch;
  k.e1 = (uint32_t)(epoch >> 32);
  return k;
}

ppo::LossHp loss_hp(const auv_ppo* p) {
  const auv_ppo_config& c = p->cfg;
  return {c.clip_eps, c.vf_coef, c.ent_coef, c.logstd_min, c.logstd_max, (int)c.norm_adv};
}

// C = op(A) op(B) in column-major terms (ta / tb: the operand is
// transposed), A and B in the activation type, C in that type too (c32 =
// false) or fp32 (c32 = true): the library's GEMM (k_gemm.cu) on the
// row-major product C'[n][m] = sum_k opB(k, n) opA(m, k), whose first
// operand is B (K-major unless transposed) and second A (K-major when
// transposed).
cudaError_t gemm(auv_ppo* p, bool ta, bool tb, int m, int n, int k, const void* A, int lda,
                 const void* B, int ldb, void* C, int ldc, bool c32, cudaStream_t s) {
  const auv::gemm::Operand a = {B, ldb, tb}, b = {A, lda, !ta};
  return auv::gemm::launch(static_cast<auv::gemm::Prec>(p->cfg.precision), n, m, k, a, b, C, ldc,
                           p->bf16 && !c32, 0.0f, p->gws, p->gws_bytes, p->st, s);
}

// Workspace of every product the learner runs (both networks).
size_t gemm_workspace(const ppo::Dims& d, const int out[2]) {
  size_t b = 0;
  for (int k = 0; k < 2; ++k) {
    const int o = out[k];
    const int shapes[8][3] = {{d.B, d.H, d.Dp}, {d.B, d.H, d.Hp}, {d.B, o, d.Hp}, {o, d.Hp, d.B},
                              {d.B, d.H, o},    {d.H, d.Hp, d.B}, {d.B, d.H, d.H}, {d.H, d.Dp, d.B}};
    for (const auto& sh : shapes) b = std::max(b, auv::gemm::workspace_bytes(sh[0], sh[1], sh[2]));
  }
  return b;
}

size_t net_offset(const auv_ppo* p, int net) { return net ? p->n_aug[0] : 0; }

// The GEMM operand copy of network `net`'s augmented weights.
const char* weights_for_gemm(const auv_ppo* p, int net) {
  const size_t o = net_offset(p, net);
  return p->bf16 ? static_cast<const char*>(p->wb) + o * 2
                 : reinterpret_cast<const char*>(p->w + o);
}

int ld_head(const auv_ppo* p, int net) { return net ? p->d.ld_val : p->d.ld_pol; }

// Column-major view (the gemm() arguments): a sample-major [B][ld] array is an ld x B
// matrix; a row-major weight [out][in_p] is an in_p x out matrix.
//   Z1 = W1a^T X,  Z2 = W2a^T H1,  Y = W3a^T H2           (forward)
//   gW3a = H2 gY^T, gH2 = W3 gY, gW2a = H1 gZ2^T, gH1 = W2 gZ2, gW1a = X gZ1^T
int forward(auv_ppo* p, int net, cudaStream_t s) {
  const ppo::Dims& d = p->d;
  const size_t es = p->esz;
  const char* w = weights_for_gemm(p, net);
  const char *w1 = w, *w2 = w + (size_t)d.H * d.Dp * es, *w3 = w2 + (size_t)d.H * d.Hp * es;
  cudaError_t e;
  if ((e = gemm(p, true, false, d.H, d.B, d.Dp, w1, d.Dp, p->X, d.Dp, p->h1[net],
                 d.Ha, false, s)))
    return cuda_fail(p, e, "forward layer 1");
  if ((e = ppo::launch_tanh_fwd(p->bf16, p->h1[net], d.Ha, d.B, d.H, s)))
    return cuda_fail(p, e, "tanh 1");
  if ((e = gemm(p, true, false, d.H, d.B, d.Hp, w2, d.Hp, p->h1[net], d.Ha,
                 p->h2[net], d.Ha, false, s)))
    return cuda_fail(p, e, "forward layer 2");
  if ((e = ppo::launch_tanh_fwd(p->bf16, p->h2[net], d.Ha, d.B, d.H, s)))
    return cuda_fail(p, e, "tanh 2");
  if ((e = gemm(p, true, false, p->out[net], d.B, d.Hp, w3, d.Hp, p->h2[net], d.Ha,
                 p->y[net], ld_head(p, net), true, s)))
    return cuda_fail(p, e, "forward layer 3");
  return AUV_OK;
}

int backward(auv_ppo* p, int net, const void* gy, cudaStream_t s) {
  const ppo::Dims& d = p->d;
  const size_t es = p->esz;
  const int out = p->out[net], ldy = ld_head(p, net);
  const char* w = weights_for_gemm(p, net);
  const char *w2 = w + (size_t)d.H * d.Dp * es, *w3 = w2 + (size_t)d.H * d.Hp * es;
  float* g = p->g + net_offset(p, net);
  float *g1 = g, *g2 = g + (size_t)d.H * d.Dp, *g3 = g2 + (size_t)d.H * d.Hp;
  void* gz2 = p->gb[net];
  void* gz1 = p->h2[net];       // H2 is dead once gZ2 exists
  cudaError_t e;
  if ((e = gemm(p, false, true, d.Hp, out, d.B, p->h2[net], d.Ha, gy, ldy, g3, d.Hp,
                 true, s)))
    return cuda_fail(p, e, "gradient W3");
  if (p->eng) {
    // gZ2 and gZ1 (into the dead H2) on the tensor-core engine, then the
    // weight gradients of layers 2 and 1
    if ((e = auv::launch_learn_backward_bf16(
             net ? p->img_bv : p->img_bp, out, static_cast<const uint16_t*>(gy), ldy, (size_t)d.B,
             static_cast<const uint16_t*>(p->h2[net]), static_cast<const uint16_t*>(p->h1[net]), d.Ha,
             static_cast<uint16_t*>(gz2), d.H, static_cast<uint16_t*>(gz1), d.Ha, p->st, s)))
      return cuda_fail(p, e, "engine backward");
    if ((e = gemm(p, false, true, d.Hp, d.H, d.B, p->h1[net], d.Ha, gz2, d.H, g2, d.Hp,
                   true, s)))
      return cuda_fail(p, e, "gradient W2");
    if ((e = gemm(p, false, true, d.Dp, d.H, d.B, p->X, d.Dp, gz1, d.Ha, g1, d.Dp,
                   true, s)))
      return cuda_fail(p, e, "gradient W1");
    return AUV_OK;
  }
  if ((e = gemm(p, false, false, d.H, d.B, out, w3, d.Hp, gy, ldy, gz2, d.H, false, s)))
    return cuda_fail(p, e, "gradient H2");
  if ((e = ppo::launch_tanh_bwd(p->bf16, gz2, d.H, p->h2[net], d.Ha, d.B, d.H, s)))
    return cuda_fail(p, e, "tanh' 2");
  if ((e = gemm(p, false, true, d.Hp, d.H, d.B, p->h1[net], d.Ha, gz2, d.H, g2, d.Hp,
                 true, s)))
    return cuda_fail(p, e, "gradient W2");
  if ((e = gemm(p, false, false, d.H, d.B, d.H, w2, d.Hp, gz2, d.H, gz1, d.Ha, false, s)))
    return cuda_fail(p, e, "gradient H1");
  if ((e = ppo::launch_tanh_bwd(p->bf16, gz1, d.Ha, p->h1[net], d.Ha, d.B, d.H, s)))
    return cuda_fail(p, e, "tanh' 1");
  if ((e = gemm(p, false, true, d.Dp, d.H, d.B, p->X, d.Dp, gz1, d.Ha, g1, d.Dp,
                 true, s)))
    return cuda_fail(p, e, "gradient W1");
  return AUV_OK;
}

// The step variables for the next launches on s (copied from pageable host
// memory: the call returns once the source has been staged).
int set_ctl(auv_ppo* p, uint64_t epoch0, uint32_t n_mb, uint32_t step, uint64_t t,
            cudaStream_t s) {
  const ppo::StepCtl c = {epoch0, t, n_mb, step};
  cudaError_t e = cudaMemcpyAsync(p->ctl, &c, sizeof(c), cudaMemcpyHostToDevice, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "step control");
}

int convert(auv_ppo* p, float* flat_pol, float* flat_val, float* aug, bool to_aug,
            cudaStream_t s);

int grads_impl(auv_ppo* p, const auv_ppo_batch* b, float* acc, cudaStream_t s) {
  const ppo::Dims& d = p->d;
  const uint32_t m = b->T * b->N;
  cudaError_t e =
      p->use_sm ? ppo::launch_gather_sm(d, perm_key(p, m, 0), p->ctl, p->sm_buf, p->smp, p->X, s)
                : ppo::launch_gather(d, perm_key(p, m, 0), p->ctl, b->obs, b->act, b->logp, b->adv,
                                     b->ret, b->N, p->smp, p->X, s);
  if (e != cudaSuccess) return cuda_fail(p, e, "gather");
  int rc;
  if (p->eng) {
    // Both networks on the tensor-core engine: flat fp32 weights, packed bf16
    // images, then one launch per network writing H1, H2 and the head.
    if ((rc = convert(p, p->flat_eng, p->flat_eng + p->n_flat[0], p->w, false, s))) return rc;
    if ((e = auv::launch_pack_learner_bf16(d.D, p->out[0], d.value_only ? nullptr : p->flat_eng,
                                           p->flat_eng + p->n_flat[0], p->img_p, p->img_v,
                                           p->img_bp, p->img_bv, s)))
      return cuda_fail(p, e, "pack engine weights");
    for (int net = d.value_only ? 1 : 0; net < 2; ++net) {
      if ((e = auv::launch_learn_forward_bf16(net == 0, net ? p->img_v : p->img_p, d.D, p->out[net],
                                         static_cast<const uint16_t*>(p->X), d.Dp, (size_t)d.B,
                                         static_cast<uint16_t*>(p->h1[net]),
                                         static_cast<uint16_t*>(p->h2[net]), d.Ha, p->y[net],
                                         ld_head(p, net), p->st, s)))
        return cuda_fail(p, e, "engine forward");
    }
  } else if ((!d.value_only && (rc = forward(p, 0, s))) || (rc = forward(p, 1, s))) {
    return rc;
  }
  const ppo::LossHp hp = loss_hp(p);
  if ((e = ppo::launch_head(d, hp, p->y[0], p->y[1], p->smp, p->g_y, p->g_v, p->head_part, s)))
    return cuda_fail(p, e, "loss head");
  if ((e = ppo::launch_stats(d, hp, p->head_part, p->mb, acc, s))) return cuda_fail(p, e, "statistics");
  if ((!d.value_only && (rc = backward(p, 0, p->g_y, s))) || (rc = backward(p, 1, p->g_v, s)))
    return rc;
  return AUV_OK;
}

// Adam step t + 1 with t from the step control (the caller advances p->t).
int apply_impl(auv_ppo* p, float* acc, cudaStream_t s) {
  const auv_ppo_config& c = p->cfg;
  ppo::AdamHp hp;
  hp.lr = c.lr;
  hp.b1 = c.adam_beta1;
  hp.b2 = c.adam_beta2;
  hp.eps = c.adam_eps;
  hp.max_norm = c.max_grad_norm;
  cudaError_t e = ppo::launch_adam(p->w, p->g, p->m, p->v, p->n_aug_all, p->norm_part, hp, p->ctl,
                                   p->mb, acc, p->wb, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "Adam");
}

// One whole gradient step of an update (gather .. Adam, then the step
// control advances), captured once per batch into p->step_graph on the
// private stream.  On any capture failure the update launches directly.
bool same_batch(const auv_ppo_batch& a, const auv_ppo_batch& b) {
  return a.obs == b.obs && a.act == b.act && a.logp == b.logp && a.adv == b.adv &&
         a.ret == b.ret && a.T == b.T && a.N == b.N;
}

void drop_graph(auv_ppo* p) {
  if (p->step_graph) cudaGraphExecDestroy(p->step_graph);
  p->step_graph = nullptr;
}

bool capture_step(auv_ppo* p, const auv_ppo_batch* b) {
  drop_graph(p);
  if (!p->gstream &&
      (cudaStreamCreateWithFlags(&p->gstream, cudaStreamNonBlocking) != cudaSuccess ||
       cudaEventCreateWithFlags(&p->ev_in, cudaEventDisableTiming) != cudaSuccess ||
       cudaEventCreateWithFlags(&p->ev_out, cudaEventDisableTiming) != cudaSuccess))
    return false;
  if (cudaStreamBeginCapture(p->gstream, cudaStreamCaptureModeThreadLocal) != cudaSuccess)
    return false;
  const bool ok = grads_impl(p, b, p->acc, p->gstream) == AUV_OK &&
                  apply_impl(p, p->acc, p->gstream) == AUV_OK &&
                  ppo::launch_step_advance(p->ctl, p->gstream) == cudaSuccess;
  cudaGraph_t g = nullptr;
  const cudaError_t e = cudaStreamEndCapture(p->gstream, &g);
  bool done = ok && e == cudaSuccess && g &&
              cudaGraphInstantiate(&p->step_graph, g, 0) == cudaSuccess;
  if (g) cudaGraphDestroy(g);
  if (!done) {
    p->step_graph = nullptr;
    cudaGetLastError();
    return false;
  }
  p->graph_batch = *b;
  p->graph_sm = p->use_sm ? p->sm_buf : nullptr;
  return true;
}

// Convert both networks between a caller's flat parameter vector (device
// memory) and an augmented learner vector.
int convert(auv_ppo* p, float* flat_pol, float* flat_val, float* aug, bool to_aug,
            cudaStream_t s) {
  const ppo::Dims& d = p->d;
  const cudaError_t e = ppo::launch_convert_pair(flat_pol, aug, p->out[0], flat_val, aug + p->n_aug[0],
                                                 p->out[1], d.D, d.Dp, d.H, d.Hp, to_aug, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "weight layout conversion");
}

// Copy a caller's policy/value pair (device or host) into the flat staging
// vector, then into the augmented vector dst.
int load_pair(auv_ppo* p, const float* pol, const float* val, float* dst, cudaStream_t s) {
  cudaError_t e = cudaMemcpyAsync(p->flat, pol, p->n_flat[0] * 4, cudaMemcpyDefault, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(p->flat + p->n_flat[0], val, p->n_flat[1] * 4, cudaMemcpyDefault, s);
  if (e != cudaSuccess) return cuda_fail(p, e, "copy in");
  int rc = convert(p, p->flat, p->flat + p->n_flat[0], dst, true, s);
  if (rc) return rc;
  if (dst == p->w && p->bf16 && (e = ppo::launch_to_bf16(p->w, p->wb, p->n_aug_all, s)))
    return cuda_fail(p, e, "bf16 weight copy");
  e = cudaStreamSynchronize(s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "synchronise");
}

int store_pair(auv_ppo* p, float* src, float* pol, float* val, cudaStream_t s) {
  int rc = convert(p, p->flat, p->flat + p->n_flat[0], src, false, s);
  if (rc) return rc;
  cudaError_t e = cudaMemcpyAsync(pol, p->flat, p->n_flat[0] * 4, cudaMemcpyDefault, s);
  if (e == cudaSuccess)
    e = cudaMemcpyAsync(val, p->flat + p->n_flat[0], p->n_flat[1] * 4, cudaMemcpyDefault, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "copy out");
}

}  // namespace

extern "C" {

const char* ppo_last_error(const auv_ppo* p) { return p ? p->err : g_err; }

int ppo_create(const auv_ppo_config* cfg, auv_ppo** out) {
  if (!out) return fail(nullptr, AUV_ERR_INVALID, "out is NULL");
  *out = nullptr;
  int rc = validate(cfg);
  if (rc) return rc;
  auv_ppo* p = new (std::nothrow) auv_ppo();
  if (!p) return fail(nullptr, AUV_ERR_INVALID, "out of host memory");
  p->cfg = *cfg;
  cudaGetDevice(&p->device);
  ppo::Dims& d = p->d;
  d.D = (int)cfg->obs_dim;
  d.Dp = round8(d.D + 1);     // rows of 16-byte multiples in fp32 and bf16
  d.A = (int)cfg->act_dim;
  d.H = (int)cfg->hidden;
  d.Hp = round8(d.H + 1);
  d.B = (int)cfg->minibatch;
  d.ld_pol = round8(2 * d.A);
  d.ld_val = 8;
  d.bf16 = cfg->precision == AUV_PPO_BF16;
  d.Ha = d.bf16 ? (d.H + 16) / 16 * 16 : d.Hp;
  d.value_only = (cfg->flags & AUV_PPO_VALUE_ONLY) ? 1 : 0;
  p->bf16 = d.bf16 != 0;
  p->esz = p->bf16 ? 2 : 4;
  p->out[0] = 2 * d.A;
  p->out[1] = 1;
  for (int k = 0; k < 2; ++k) {
    const size_t o = (size_t)p->out[k];
    p->n_flat[k] = (size_t)d.H * d.D + d.H + (size_t)d.H * d.H + d.H + o * d.H + o;
    p->n_aug[k] = ppo::aug_count(d.D, d.Dp, d.H, d.Hp, p->out[k]);
  }
  p->n_aug_all = p->n_aug[0] + p->n_aug[1];
  // the engine's networks: hidden 256, input <= 18, head <= 16 (2A <= 16)
  p->eng = p->bf16 && d.H == 256 && d.D <= auv::kObs && !(cfg->flags & AUV_PPO_GEMM_PATH);
  const size_t gws_bytes = gemm_workspace(d, p->out);
  // one allocation, 256-byte aligned pieces
  const size_t B = (size_t)d.B, nb = (B + 255) / 256;
  size_t off = 0;
  auto take = [&](size_t bytes) {
    const size_t o = off;
    off += (bytes + 255) & ~(size_t)255;
    return o;
  };
  const size_t es = p->esz;
  const size_t o_w = take(p->n_aug_all * 4), o_g = take(p->n_aug_all * 4),
               o_m = take(p->n_aug_all * 4), o_v = take(p->n_aug_all * 4),
               o_wb = take(p->bf16 ? p->n_aug_all * 2 : 0),
               o_flat = take((p->n_flat[0] + p->n_flat[1]) * 4), o_x = take(B * d.Dp * es),
               o_act = take(B * d.A * 4), o_lp = take(B * 4), o_adv = take(B * 4),
               o_ret = take(B * 4), o_ap = take(nb * 2 * 8), o_gy = take(B * d.ld_pol * es),
               o_gv = take(B * d.ld_val * es), o_hp = take(nb * 5 * 4),
               o_np = take((ppo::kNormBlocks + 3) * 4), o_mb = take(AUV_PPO_STATS * 4),
               o_acc = take(AUV_PPO_STATS * 4), o_ctl = take(sizeof(ppo::StepCtl)),
               o_ws = take(gws_bytes),
               o_ip = take(p->eng ? auv::bf16_policy_image_bytes() : 0),
               o_iv = take(p->eng ? auv::bf16_value_image_bytes() : 0),
               o_ibp = take(p->eng ? auv::bf16_back_image_bytes() : 0),
               o_ibv = take(p->eng ? auv::bf16_back_image_bytes() : 0),
               o_fe = take(p->eng ? (p->n_flat[0] + p->n_flat[1]) * 4 : 0),
               o_st = take(sizeof(Status));
  size_t o_h1[2], o_h2[2], o_gb[2], o_y[2];
  for (int k = 0; k < 2; ++k) {
    o_h1[k] = take(B * d.Ha * es);
    o_h2[k] = take(B * d.Ha * es);
    o_gb[k] = take(B * d.H * es);
    o_y[k] = take(B * (k ? d.ld_val : d.ld_pol) * 4);
  }
  cudaError_t e = cudaMalloc(&p->mem, off);
  if (e != cudaSuccess) {
    delete p;
    return cuda_fail(nullptr, e, "cudaMalloc(learner)");
  }
  char* base = p->mem;
  p->w = reinterpret_cast<float*>(base + o_w);
  p->g = reinterpret_cast<float*>(base + o_g);
  p->m = reinterpret_cast<float*>(base + o_m);
  p->v = reinterpret_cast<float*>(base + o_v);
  p->wb = p->bf16 ? base + o_wb : nullptr;
  p->flat = reinterpret_cast<float*>(base + o_flat);
  p->X = base + o_x;
  p->smp.act = reinterpret_cast<float*>(base + o_act);
  p->smp.logp = reinterpret_cast<float*>(base + o_lp);
  p->smp.adv = reinterpret_cast<float*>(base + o_adv);
  p->smp.ret = reinterpret_cast<float*>(base + o_ret);
  p->smp.adv_part = reinterpret_cast<double*>(base + o_ap);
  p->g_y = base + o_gy;
  p->g_v = base + o_gv;
  p->head_part = reinterpret_cast<float*>(base + o_hp);
  p->norm_part = reinterpret_cast<float*>(base + o_np);
  p->mb = reinterpret_cast<float*>(base + o_mb);
  p->acc = reinterpret_cast<float*>(base + o_acc);
  p->ctl = reinterpret_cast<ppo::StepCtl*>(base + o_ctl);
  p->gws = reinterpret_cast<float*>(base + o_ws);
  p->gws_bytes = gws_bytes;
  if (p->eng) {
    p->img_p = base + o_ip;
    p->img_v = base + o_iv;
    p->img_bp = base + o_ibp;
    p->img_bv = base + o_ibv;
    p->flat_eng = reinterpret_cast<float*>(base + o_fe);
  }
  p->st = reinterpret_cast<Status*>(base + o_st);
  for (int k = 0; k < 2; ++k) {
    p->h1[k] = base + o_h1[k];
    p->h2[k] = base + o_h2[k];
    p->gb[k] = base + o_gb[k];
    p->y[k] = reinterpret_cast<float*>(base + o_y[k]);
  }
  e = cudaMemset(p->mem, 0, off);
  if (e == cudaSuccess) {
    const Status s0 = {0, 0, INT32_MAX, 0};
    e = cudaMemcpy(p->st, &s0, sizeof(s0), cudaMemcpyHostToDevice);
  }
  for (int k = 0; k < 2 && e == cudaSuccess; ++k) {
    e = ppo::launch_fill_ones(p->bf16, p->h1[k], d.Ha, d.H, d.B, 0);
    if (e == cudaSuccess) e = ppo::launch_fill_ones(p->bf16, p->h2[k], d.Ha, d.H, d.B, 0);
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaFree(p->mem);
    delete p;
    return cuda_fail(nullptr, e, "initialise learner memory");
  }
  *out = p;
  return AUV_OK;
}

int ppo_destroy(auv_ppo* p) {
  if (!p) return AUV_ERR_INVALID;
  int prev = -1;
  cudaGetDevice(&prev);
  cudaSetDevice(p->device);
  cudaDeviceSynchronize();
  drop_graph(p);
  if (p->ev_in) cudaEventDestroy(p->ev_in);
  if (p->ev_out) cudaEventDestroy(p->ev_out);
  if (p->gstream) cudaStreamDestroy(p->gstream);
  if (p->sm_buf) cudaFree(p->sm_buf);
  cudaFree(p->mem);
  if (prev >= 0) cudaSetDevice(prev);
  delete p;
  return AUV_OK;
}

int ppo_param_counts(const auv_ppo* p, uint64_t* n_policy, uint64_t* n_value) {
  if (!p || !n_policy || !n_value) return AUV_ERR_INVALID;
  *n_policy = p->n_flat[0];
  *n_value = p->n_flat[1];
  return AUV_OK;
}

int ppo_set_weights(auv_ppo* p, const float* policy, const float* value, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  if (!policy || !value) return fail(p, AUV_ERR_INVALID, "weights are NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t bytes = p->n_aug_all * 4;
  cudaError_t e = cudaMemsetAsync(p->m, 0, bytes, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(p->v, 0, bytes, s);
  if (e != cudaSuccess) return cuda_fail(p, e, "clear Adam moments");
  if ((rc = load_pair(p, policy, value, p->w, s))) return rc;
  p->t = 0;
  p->epoch = 0;
  return AUV_OK;
}

int ppo_get_weights(auv_ppo* p, float* policy, float* value, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  if (!policy || !value) return fail(p, AUV_ERR_INVALID, "outputs are NULL");
  return store_pair(p, p->w, policy, value, static_cast<cudaStream_t>(stream));
}

int ppo_export_weights(auv_ppo* p, float* policy, float* value, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc || (rc = check_dev(p, policy, "policy")) || (rc = check_dev(p, value, "value"))) return rc;
  return convert(p, policy, value, p->w, false, static_cast<cudaStream_t>(stream));
}

int ppo_get_state(auv_ppo* p, float* m, float* v, uint64_t* t, uint64_t* epoch, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  if (!m || !v || !t || !epoch) return fail(p, AUV_ERR_INVALID, "outputs are NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = store_pair(p, p->m, m, m + p->n_flat[0], s))) return rc;
  if ((rc = store_pair(p, p->v, v, v + p->n_flat[0], s))) return rc;
  *t = p->t;
  *epoch = p->epoch;
  return AUV_OK;
}

int ppo_set_state(auv_ppo* p, const float* m, const float* v, uint64_t t, uint64_t epoch,
                  void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  if (!m || !v) return fail(p, AUV_ERR_INVALID, "moments are NULL");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = load_pair(p, m, m + p->n_flat[0], p->m, s))) return rc;
  if ((rc = load_pair(p, v, v + p->n_flat[0], p->v, s))) return rc;
  p->t = t;
  p->epoch = epoch;
  return AUV_OK;
}

int ppo_grads(auv_ppo* p, const auv_ppo_batch* batch, uint64_t epoch, uint32_t minibatch,
              float* grad, float* stats, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc || (rc = check_batch(p, batch))) return rc;
  if (((uint64_t)minibatch + 1) * p->d.B > (uint64_t)batch->T * batch->N)
    return fail(p, AUV_ERR_SIZE, "minibatch %u needs %llu rows, the batch has %llu", minibatch,
                (unsigned long long)(((uint64_t)minibatch + 1) * p->d.B),
                (unsigned long long)batch->T * batch->N);
  if (grad && (rc = check_dev(p, grad, "grad"))) return rc;
  if (stats && (rc = check_dev(p, stats, "stats"))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if ((rc = set_ctl(p, epoch, 1u << 31, minibatch, p->t, s))) return rc;
  if ((rc = grads_impl(p, batch, nullptr, s))) return rc;
  if (grad && (rc = convert(p, grad, grad + p->n_flat[0], p->g, false, s))) return rc;
  if (stats) {
    cudaError_t e = cudaMemcpyAsync(stats, p->mb, AUV_PPO_STATS * 4, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(p, e, "copy statistics");
  }
  return AUV_OK;
}

int ppo_apply(auv_ppo* p, const float* grad, float* stats, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  if (grad && (rc = check_dev(p, grad, "grad"))) return rc;
  if (stats && (rc = check_dev(p, stats, "stats"))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (grad) {
    cudaError_t e = cudaMemcpyAsync(p->flat, grad, (p->n_flat[0] + p->n_flat[1]) * 4,
                                    cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(p, e, "copy gradient");
    if ((rc = convert(p, p->flat, p->flat + p->n_flat[0], p->g, true, s))) return rc;
  }
  if ((rc = set_ctl(p, p->epoch, 1u << 31, 0, p->t, s))) return rc;
  if ((rc = apply_impl(p, nullptr, s))) return rc;
  p->t += 1;
  if (stats) {
    cudaError_t e = cudaMemcpyAsync(stats + 5, p->mb + 5, 4, cudaMemcpyDeviceToDevice, s);
    if (e != cudaSuccess) return cuda_fail(p, e, "copy gradient norm");
  }
  return AUV_OK;
}

int ppo_status(auv_ppo* p, auv_status* out, void* stream) {
  if (!p || !out) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  Status h;
  cudaError_t e = cudaMemcpyAsync(&h, p->st, sizeof(h), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(p, e, "read status");
  out->code = h.code;
  out->nan_flag = h.nan_flag;
  out->first_nan_env = h.first_nan_env == INT32_MAX ? -1 : h.first_nan_env;
  out->timeouts = h.timeouts;
  if (h.code != 0) fail(p, h.code, "device status %d (timeouts %d)", h.code, h.timeouts);
  return h.code;
}

int ppo_clear_status(auv_ppo* p, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc) return rc;
  static const Status s0 = {0, 0, INT32_MAX, 0};
  cudaError_t e = cudaMemcpyAsync(p->st, &s0, sizeof(s0), cudaMemcpyHostToDevice,
                                  static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(p, e, "clear status");
}

int ppo_update(auv_ppo* p, const auv_ppo_batch* batch, uint32_t epochs, uint32_t n_minibatches,
               float* stats, void* stream) {
  if (!p) return AUV_ERR_INVALID;
  int rc = check_device(p);
  if (rc || (rc = check_batch(p, batch))) return rc;
  if (epochs < 1 || n_minibatches < 1) return fail(p, AUV_ERR_INVALID, "epochs and n_minibatches must be >= 1");
  if ((uint64_t)n_minibatches * p->d.B > (uint64_t)batch->T * batch->N)
    return fail(p, AUV_ERR_SIZE, "%u minibatches of %d exceed the batch's %llu rows", n_minibatches,
                p->d.B, (unsigned long long)batch->T * batch->N);
  if (stats && (rc = check_dev(p, stats, "stats"))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint64_t steps = (uint64_t)epochs * n_minibatches;
  // The sample-major copy: grown when a larger batch arrives (cudaFree waits
  // for the work that may still read the old one); without it the steps
  // gather from the batch's own arrays.
  const size_t rows = (size_t)batch->T * batch->N;
  const int ws = ppo::sample_row_floats(p->d.D, p->d.A);
  if (p->sm_rows < rows) {
    if (p->sm_buf) cudaFree(p->sm_buf);
    p->sm_buf = nullptr;
    p->sm_rows = 0;
    if (cudaMalloc(&p->sm_buf, rows * ws * sizeof(float)) == cudaSuccess) p->sm_rows = rows;
    else p->sm_buf = nullptr;
    cudaGetLastError();
  }
  p->use_sm = p->sm_buf != nullptr;
  struct SmScope {   // the copy serves this update's steps only (ppo_grads gathers directly)
    auv_ppo* q;
    ~SmScope() { q->use_sm = false; }
  } sm_scope{p};
  // replay the captured step on the private stream when it can be had
  if (!p->graph_failed &&
      (!p->step_graph || !same_batch(p->graph_batch, *batch) ||
       p->graph_sm != (p->use_sm ? p->sm_buf : nullptr)) &&
      !capture_step(p, batch))
    p->graph_failed = true;
  const bool graph = p->step_graph != nullptr && !p->graph_failed;
  cudaStream_t r = s;
  cudaError_t e;
  if (graph) {
    if ((e = cudaEventRecord(p->ev_in, s)) || (e = cudaStreamWaitEvent(p->gstream, p->ev_in, 0)))
      return cuda_fail(p, e, "order update after caller");
    r = p->gstream;
  }
  if ((rc = set_ctl(p, p->epoch, n_minibatches, 0, p->t, r))) return rc;
  if ((e = cudaMemsetAsync(p->acc, 0, AUV_PPO_STATS * 4, r)))
    return cuda_fail(p, e, "clear statistics");
  if (p->use_sm && (e = ppo::launch_transpose_batch(p->d.D, p->d.A, batch->T, batch->N, batch->obs,
                                                     p->d.value_only ? nullptr : batch->act,
                                                     p->d.value_only ? nullptr : batch->logp,
                                                     p->d.value_only ? nullptr : batch->adv,
                                                     batch->ret, p->sm_buf, r)))
    return cuda_fail(p, e, "sample-major batch copy");
  for (uint64_t k = 0; k < steps; ++k) {
    if (graph) {
      if ((e = cudaGraphLaunch(p->step_graph, r))) return cuda_fail(p, e, "launch step graph");
    } else {
      if ((rc = grads_impl(p, batch, p->acc, r)) || (rc = apply_impl(p, p->acc, r))) return rc;
      if ((e = ppo::launch_step_advance(p->ctl, r))) return cuda_fail(p, e, "advance step");
    }
  }
  if (stats && (e = ppo::launch_finish(p->acc, stats, r)) != cudaSuccess)
    return cuda_fail(p, e, "statistics");
  if (graph && ((e = cudaEventRecord(p->ev_out, r)) || (e = cudaStreamWaitEvent(s, p->ev_out, 0))))
    return cuda_fail(p, e, "order caller after update");
  p->t += steps;
  p->epoch += epochs;
  return AUV_OK;
}

}  // extern "C"
