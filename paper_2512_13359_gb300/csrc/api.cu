// api.cu -- the extern "C" entry points of libauvenv.so (include/auvenv.h):
// argument and configuration validation, the library workspace, and the
// dispatch of each call to its kernels on the caller's stream.
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>


#include "auv_kernels.h"
#include "auv_bf16.h"
#include "auvenv.h"

using auv::Buffers;
using auv::Model;
using auv::Status;
using auv::Traj;

struct auv_env {
  auv_config cfg;
  Model model;
  Buffers buf;
  int device;
  uint64_t t_g;
  char* workspace;          // device: [status | policy weights | value weights | staging]
  Status* status;
  float* w_policy_f32;      // fp32 mode: row-major weights as given
  float* w_value_f32;
  void* w_policy_packed;    // bf16 mode: packed operand images
  void* w_value_packed;
  float* staging;           // fp32 copy of the caller's weights (bf16 mode)
  size_t policy_count, value_count;
  bool weights_set;
  char err[256];
  // Host trajectories (env_rollout): two device segment buffers, the copy
  // stream that drains them, and the events ordering the two; made on first use.
  char* stage = nullptr;
  size_t stage_bytes = 0;
  cudaStream_t copy_stream = nullptr;
  cudaEvent_t seg_done[2] = {nullptr, nullptr};
  cudaEvent_t copy_done[2] = {nullptr, nullptr};
  int last_copy = -1;       // buffer whose copy_done ends the last staged call
  // Adjoint windows (env_adjoint): per-step inputs of the forward pass.
  float* adj_scratch = nullptr;
  size_t adj_scratch_floats = 0;
  // Inverse allocation (env_inverse_allocate): made on first use.
  bool inv_ready = false;
  auv::InvAlloc inv;
  // SHAC windows (env_shac_window): workspace for the last (N, T, H), made on
  // first use.
  char* shac_ws = nullptr;
  size_t shac_ws_bytes = 0;
  int shac_T = 0;
};

namespace {

thread_local char g_create_err[256] = "";

int fail(auv_env* env, int code, const char* fmt, ...) {
  char* dst = env ? env->err : g_create_err;
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(dst, 256, fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(auv_env* env, cudaError_t e, const char* what) {
  return fail(env, AUV_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

size_t mlp_count(size_t in, size_t H, size_t out) {
  return H * in + H + H * H + H + out * H + out;
}

bool is_paper(const auv_config* c) { return c->model == AUV_MODEL_PAPER; }
size_t obs_dim(const auv_config* c) { return is_paper(c) ? AUV_PAPER_OBS_DIM : AUV_OBS_DIM; }
size_t act_dim(const auv_config* c) { return is_paper(c) ? AUV_PAPER_ACT_DIM : AUV_ACT_DIM; }

bool finite_pos(float x) { return std::isfinite(x) && x > 0.0f; }
bool finite_nonneg(float x) { return std::isfinite(x) && x >= 0.0f; }

enum PtrKind { kBad, kDevice, kHostMapped };

// Classifies a pointer and returns the address a kernel must use.
PtrKind classify(const void* p, void** dev) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return kBad;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) {
    *dev = const_cast<void*>(p);
    return kDevice;
  }
  if (a.type == cudaMemoryTypeHost && a.devicePointer) {
    *dev = a.devicePointer;
    return kHostMapped;
  }
  return kBad;
}

int check_device_buffer(auv_env* env, const void* p, const char* name, size_t align) {
  void* d = nullptr;
  if (!p) return fail(env, AUV_ERR_INVALID, "%s is NULL", name);
  if (reinterpret_cast<uintptr_t>(p) % align)
    return fail(env, AUV_ERR_SIZE, "%s is not %zu-byte aligned", name, align);
  if (classify(p, &d) != kDevice) return fail(env, AUV_ERR_SIZE, "%s is not device memory", name);
  return AUV_OK;
}

// Output buffer: device memory or mapped page-locked host memory.
int map_output(auv_env* env, void* p, const char* name, size_t align, void** dev) {
  *dev = nullptr;
  if (!p) return AUV_OK;
  if (reinterpret_cast<uintptr_t>(p) % align)
    return fail(env, AUV_ERR_SIZE, "%s is not %zu-byte aligned", name, align);
  if (classify(p, dev) == kBad)
    return fail(env, AUV_ERR_SIZE, "%s is neither device memory nor mapped page-locked host memory",
                name);
  return AUV_OK;
}

// Shared network and episode checks (both models).
int validate_networks(const auv_config* c, uint32_t out_mean) {
  if (c->policy_out != out_mean && c->policy_out != 2 * out_mean)
    return fail(nullptr, AUV_ERR_INVALID, "policy_out must be %u or %u", out_mean, 2 * out_mean);
  if (c->mlp_mode != AUV_MLP_FP32 && c->mlp_mode != AUV_MLP_BF16 && c->mlp_mode != AUV_MLP_TF32)
    return fail(nullptr, AUV_ERR_INVALID, "unknown mlp_mode %u", c->mlp_mode);
  if (c->has_value > 1) return fail(nullptr, AUV_ERR_INVALID, "has_value must be 0 or 1");
  if (!(c->logstd_min <= c->logstd_max) || !std::isfinite(c->logstd_min) ||
      !std::isfinite(c->logstd_max))
    return fail(nullptr, AUV_ERR_INVALID, "logstd clamp invalid");
  for (int k = 0; k < 8; ++k)
    if (!std::isfinite(c->logstd_fixed[k]))
      return fail(nullptr, AUV_ERR_INVALID, "logstd_fixed not finite");
  if (c->mlp_mode == AUV_MLP_FP32 && c->hidden != 64 && c->hidden != 256)
    return fail(nullptr, AUV_ERR_UNSUPPORTED, "fp32 networks are built for hidden 64 or 256");
  if (c->mlp_mode == AUV_MLP_TF32 &&
      (c->model != AUV_MODEL_FOSSEN || c->hidden != 256 || c->has_value))
    return fail(nullptr, AUV_ERR_UNSUPPORTED,
                "tf32 networks are built for the Fossen model, hidden 256, no value network");
  if (c->mlp_mode == AUV_MLP_BF16 && (c->hidden != 256 || c->policy_out != 2 * out_mean))
    return fail(nullptr, AUV_ERR_UNSUPPORTED,
                "bf16 networks are built for hidden 256 with the mean + log-std head");
  return AUV_OK;
}

// The paper model's own fields (the Fossen-only fields are ignored).
int validate_paper(const auv_config* c) {
  const float pi = 3.14159274f;
  if (!finite_nonneg(c->f_max) || !finite_nonneg(c->tau_max))
    return fail(nullptr, AUV_ERR_INVALID, "f_max and tau_max must be finite and >= 0");
  if (!finite_nonneg(c->fluid_density) || !finite_nonneg(c->fluid_viscosity))
    return fail(nullptr, AUV_ERR_INVALID, "fluid density and viscosity must be finite and >= 0");
  const double I0 = c->inertia[0], I1 = c->inertia[1], I2 = c->inertia[2];
  if (!(I1 + I2 > I0 && I0 + I2 > I1 && I0 + I1 > I2))
    return fail(nullptr, AUV_ERR_INVALID,
                "inertia violates the triangle inequality (no equivalent inertia box)");
  if (!std::isfinite(c->g_eff) || !finite_nonneg(c->dr_gravity_range))
    return fail(nullptr, AUV_ERR_INVALID, "effective gravity and its range must be finite");
  if (!finite_nonneg(c->init_pos_range) || !finite_nonneg(c->goal_pos_range) ||
      !finite_nonneg(c->init_att_range) || !finite_nonneg(c->goal_att_range) ||
      c->init_att_range > pi || c->goal_att_range > pi)
    return fail(nullptr, AUV_ERR_INVALID,
                "ranges must be finite and >= 0; attitude ranges <= pi");
  if (c->dr_enable > 1) return fail(nullptr, AUV_ERR_INVALID, "dr_enable must be 0 or 1");
  if (!std::isfinite(c->w_pos) || !std::isfinite(c->w_att) || !std::isfinite(c->w_act) ||
      !std::isfinite(c->w_vel) || !std::isfinite(c->w_mavg) || !std::isfinite(c->w_axes[0]) ||
      !std::isfinite(c->w_axes[1]) || !std::isfinite(c->w_axes[2]))
    return fail(nullptr, AUV_ERR_INVALID, "reward weights not finite");
  if (c->mavg_len < 1 || c->mavg_len > AUV_PAPER_HIST)
    return fail(nullptr, AUV_ERR_INVALID, "mavg_len %u outside [1, %d]", c->mavg_len,
                AUV_PAPER_HIST);
  return validate_networks(c, AUV_PAPER_ACT_DIM);
}

int validate_config(const auv_config* c) {
  if (!c) return fail(nullptr, AUV_ERR_INVALID, "cfg is NULL");
  if (c->struct_size != sizeof(auv_config))
    return fail(nullptr, AUV_ERR_INVALID, "cfg->struct_size %u != sizeof(auv_config) %zu",
                c->struct_size, sizeof(auv_config));
  if (c->n_envs < 1 || c->n_envs > (1u << 30))
    return fail(nullptr, AUV_ERR_INVALID, "n_envs %u outside [1, 2^30]", c->n_envs);
  if ((uint64_t)c->env_id_base + c->n_envs > (1ull << 32))
    return fail(nullptr, AUV_ERR_INVALID, "env_id_base + n_envs exceeds 2^32");
  if (c->substeps < 1 || c->substeps > 64)
    return fail(nullptr, AUV_ERR_INVALID, "substeps %u outside [1, 64]", c->substeps);
  if (c->episode_len < 1 || c->episode_len > (uint32_t)INT_MAX)
    return fail(nullptr, AUV_ERR_INVALID, "episode_len %u invalid", c->episode_len);
  if (!finite_pos(c->dt)) return fail(nullptr, AUV_ERR_INVALID, "dt must be finite and > 0");
  if (!finite_pos(c->mass)) return fail(nullptr, AUV_ERR_INVALID, "mass must be > 0");
  for (int k = 0; k < 3; ++k)
    if (!finite_pos(c->inertia[k])) return fail(nullptr, AUV_ERR_INVALID, "inertia must be > 0");
  if (c->model != AUV_MODEL_FOSSEN && c->model != AUV_MODEL_PAPER)
    return fail(nullptr, AUV_ERR_INVALID, "unknown model %u", c->model);
  if (is_paper(c)) return validate_paper(c);
  for (int k = 0; k < 6; ++k) {
    if (!finite_nonneg(c->added_mass[k]) || !finite_nonneg(c->damp_lin[k]) ||
        !finite_nonneg(c->damp_quad[k]))
      return fail(nullptr, AUV_ERR_INVALID, "added mass and damping must be finite and >= 0");
  }
  for (int k = 0; k < 3; ++k)
    if (!std::isfinite(c->gravity[k])) return fail(nullptr, AUV_ERR_INVALID, "gravity not finite");
  if (!finite_nonneg(c->thrust_max)) return fail(nullptr, AUV_ERR_INVALID, "thrust_max invalid");
  for (int k = 0; k < 48; ++k)
    if (!std::isfinite(c->alloc[k])) return fail(nullptr, AUV_ERR_INVALID, "alloc not finite");
  const float pi = 3.14159274f;
  if (!finite_nonneg(c->init_pos_range) || !finite_nonneg(c->goal_pos_range) ||
      !finite_nonneg(c->current_range) || !finite_nonneg(c->init_att_range) ||
      !finite_nonneg(c->goal_yaw_range) || c->init_att_range > pi || c->goal_yaw_range > pi)
    return fail(nullptr, AUV_ERR_INVALID,
                "ranges must be finite and >= 0; attitude and goal-yaw ranges <= pi");
  if (c->dr_enable > 1) return fail(nullptr, AUV_ERR_INVALID, "dr_enable must be 0 or 1");
  if (c->dr_enable) {
    if (!finite_pos(c->dr_scale_lo) || !(c->dr_scale_hi >= c->dr_scale_lo) ||
        !std::isfinite(c->dr_scale_hi) || !finite_nonneg(c->dr_buoy_range) ||
        !finite_nonneg(c->dr_cob_range))
      return fail(nullptr, AUV_ERR_INVALID, "domain-randomisation ranges invalid");
  }
  if (!std::isfinite(c->w_pos) || !std::isfinite(c->w_att) || !std::isfinite(c->w_act) ||
      !std::isfinite(c->w_vs))
    return fail(nullptr, AUV_ERR_INVALID, "reward weights not finite");
  return validate_networks(c, AUV_ACT_DIM);
}

Model build_model(const auv_config* c) {
  Model M;
  std::memset(&M, 0, sizeof(M));
  M.n = (int)c->n_envs;
  M.substeps = (int)c->substeps;
  M.episode_len = (int)c->episode_len;
  M.seed = c->seed;
  M.id_base = c->env_id_base;
  M.dr_enable = (int)c->dr_enable;
  M.policy_out = (int)c->policy_out;
  M.has_value = (int)c->has_value;
  M.hidden = (int)c->hidden;
  M.h = c->dt / (float)c->substeps;
  M.mass = c->mass;
  for (int k = 0; k < 3; ++k) M.inertia[k] = c->inertia[k];
  for (int k = 0; k < 6; ++k) {
    M.added[k] = c->added_mass[k];
    M.dlin[k] = c->damp_lin[k];
    M.dquad[k] = c->damp_quad[k];
  }
  const double g0 = c->gravity[0], g1 = c->gravity[1], g2 = c->gravity[2];
  const double gn = std::sqrt(g0 * g0 + g1 * g1 + g2 * g2);
  M.gnorm = (float)gn;
  if (gn > 0) {
    M.ghat[0] = (float)(g0 / gn);
    M.ghat[1] = (float)(g1 / gn);
    M.ghat[2] = (float)(g2 / gn);
  }
  for (int k = 0; k < 48; ++k) M.alloc_t[k] = c->alloc[k] * c->thrust_max;
  M.w_pos = c->w_pos; M.w_att = c->w_att; M.w_act = c->w_act; M.w_vs = c->w_vs;
  M.init_pos_range = c->init_pos_range;
  M.init_att_range = c->init_att_range;
  M.goal_pos_range = c->goal_pos_range;
  M.goal_yaw_range = c->goal_yaw_range;
  M.current_range = c->current_range;
  M.dr_lo = c->dr_scale_lo; M.dr_hi = c->dr_scale_hi;
  M.dr_buoy = c->dr_buoy_range; M.dr_cob = c->dr_cob_range;
  for (int k = 0; k < 8; ++k) M.logstd_fixed[k] = c->logstd_fixed[k];
  M.logstd_min = c->logstd_min; M.logstd_max = c->logstd_max;
  M.model = (int)c->model;
  if (is_paper(c)) {
    // inertia box: the uniform box with the body's mass and principal moments
    const double m = c->mass, I0 = c->inertia[0], I1 = c->inertia[1], I2 = c->inertia[2];
    const double b[3] = {std::sqrt(6 * (I1 + I2 - I0) / m), std::sqrt(6 * (I0 + I2 - I1) / m),
                         std::sqrt(6 * (I0 + I1 - I2) / m)};
    const double rho = c->fluid_density, mu = c->fluid_viscosity, pi = 3.14159265358979323846;
    const double d = (b[0] + b[1] + b[2]) / 3;
    for (int k = 0; k < 3; ++k) {
      const int j = (k + 1) % 3, l = (k + 2) % 3;
      M.kf_drag[k] = (float)(0.5 * rho * b[j] * b[l]);
      M.kt_drag[k] = (float)(rho / 64 * b[k] * (std::pow(b[j], 4) + std::pow(b[l], 4)));
      M.inv_inertia[k] = (float)(1.0 / c->inertia[k]);
      M.w_axes[k] = c->w_axes[k];
    }
    M.c_visc_f = (float)(3 * pi * mu * d);
    M.c_visc_t = (float)(pi * mu * d * d * d);
    M.inv_mass = (float)(1.0 / m);
    M.f_max = c->f_max;
    M.tau_max = c->tau_max;
    M.g_eff0 = c->g_eff;
    M.dr_grav = c->dr_gravity_range;
    M.goal_att_range = c->goal_att_range;
    M.w_vel = c->w_vel;
    M.w_mavg = c->w_mavg;
    M.mavg_len = (int)c->mavg_len;
  }
  return M;
}

int check_device(auv_env* env) {
  int cur = -1;
  cudaError_t e = cudaGetDevice(&cur);
  if (e != cudaSuccess) return cuda_fail(env, e, "cudaGetDevice");
  if (cur != env->device)
    return fail(env, AUV_ERR_INVALID, "device %d is current but the env lives on device %d", cur,
                env->device);
  return AUV_OK;
}

// Checkpoint and resume: the caller's batch arrays plus the global step.
int snapshot_arrays(auv_env* env, const auv_snapshot* snap, bool check_header) {
  if (!env || !snap) return AUV_ERR_INVALID;
  if (snap->struct_size != sizeof(auv_snapshot))
    return fail(env, AUV_ERR_INVALID, "snapshot struct_size %u != sizeof(auv_snapshot) %zu",
                snap->struct_size, sizeof(auv_snapshot));
  if (!snap->state || !snap->params || !snap->t_ep || !snap->episode)
    return fail(env, AUV_ERR_INVALID, "snapshot array is NULL");
  const void* arr[4] = {snap->state, snap->params, snap->t_ep, snap->episode};
  for (const void* p : arr)
    if (reinterpret_cast<uintptr_t>(p) % 4)
      return fail(env, AUV_ERR_SIZE, "snapshot array is not 4-byte aligned");
  if (check_header) {
    auv_layout lay;
    env_layout(env->cfg.model, &lay);
    if (snap->model != env->cfg.model || snap->n_envs != env->cfg.n_envs ||
        snap->state_fields != lay.state_fields || snap->param_fields != lay.param_fields)
      return fail(env, AUV_ERR_INVALID,
                  "snapshot (model %u, %u envs, %u/%u fields) does not match the env "
                  "(model %u, %u envs, %u/%u fields)",
                  snap->model, snap->n_envs, snap->state_fields, snap->param_fields,
                  env->cfg.model, env->cfg.n_envs, lay.state_fields, lay.param_fields);
  }
  return AUV_OK;
}

int copy_batch(auv_env* env, void* const dst[4], const void* const src[4], cudaStream_t s) {
  auv_layout lay;
  env_layout(env->cfg.model, &lay);
  const size_t n = env->cfg.n_envs;
  const size_t bytes[4] = {lay.state_fields * n * sizeof(float), lay.param_fields * n * sizeof(float),
                           n * sizeof(int32_t), n * sizeof(uint32_t)};
  for (int k = 0; k < 4; ++k) {
    cudaError_t e = cudaMemcpyAsync(dst[k], src[k], bytes[k], cudaMemcpyDefault, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "snapshot copy");
  }
  return AUV_OK;
}
}  // namespace

extern "C" {

int env_abi_version(void) { return AUV_ABI_VERSION; }

int env_layout(uint32_t model, auv_layout* out) {
  if (!out) return fail(nullptr, AUV_ERR_INVALID, "out is NULL");
  if (model == AUV_MODEL_FOSSEN) {
    *out = {AUV_OBS_DIM, AUV_ACT_DIM, AUV_STATE_FIELDS, AUV_PARAM_FIELDS};
  } else if (model == AUV_MODEL_PAPER) {
    *out = {AUV_PAPER_OBS_DIM, AUV_PAPER_ACT_DIM, AUV_PAPER_STATE_FIELDS, AUV_PAPER_PARAM_FIELDS};
  } else {
    return fail(nullptr, AUV_ERR_INVALID, "unknown model %u", model);
  }
  return AUV_OK;
}

const char* env_last_error(const auv_env* env) { return env ? env->err : g_create_err; }

int env_create(const auv_config* cfg, const auv_buffers* buf, auv_env** out) {
  g_create_err[0] = 0;
  if (!out) return fail(nullptr, AUV_ERR_INVALID, "out is NULL");
  *out = nullptr;
  int rc = validate_config(cfg);
  if (rc) return rc;
  if (!buf) return fail(nullptr, AUV_ERR_INVALID, "buf is NULL");
  if ((rc = check_device_buffer(nullptr, buf->state, "state", 16))) return rc;
  if ((rc = check_device_buffer(nullptr, buf->params, "params", 16))) return rc;
  if ((rc = check_device_buffer(nullptr, buf->t_ep, "t_ep", 16))) return rc;
  if ((rc = check_device_buffer(nullptr, buf->episode, "episode", 16))) return rc;
  auv_env* env = new (std::nothrow) auv_env;
  if (!env) return fail(nullptr, AUV_ERR_INVALID, "out of host memory");
  std::memset(env, 0, sizeof(*env));
  env->last_copy = -1;
  env->cfg = *cfg;
  env->model = build_model(cfg);
  env->buf.state = buf->state;
  env->buf.params = buf->params;
  env->buf.t_ep = buf->t_ep;
  env->buf.episode = buf->episode;
  cudaGetDevice(&env->device);
  env->policy_count = mlp_count(obs_dim(cfg), cfg->hidden, cfg->policy_out);
  env->value_count = cfg->has_value ? mlp_count(obs_dim(cfg), cfg->hidden, 1) : 0;
  // workspace: status (256 B) | fp32 policy | fp32 value | packed bf16 images
  size_t off = 256;
  const size_t pol_off = off;
  off += ((env->policy_count * 4 + 255) / 256) * 256;
  const size_t val_off = off;
  off += ((env->value_count * 4 + 255) / 256) * 256;
  size_t pol_pk_off = 0, val_pk_off = 0;
  if (cfg->mlp_mode == AUV_MLP_BF16) {
    pol_pk_off = off;
    off += ((auv::bf16_policy_image_bytes() + 1023) / 1024) * 1024;
    val_pk_off = off;
    off += ((auv::bf16_value_image_bytes() + 1023) / 1024) * 1024;
  } else if (cfg->mlp_mode == AUV_MLP_TF32) {
    pol_pk_off = off;
    off += ((auv::tf32_policy_image_bytes() + 1023) / 1024) * 1024;
  }
  cudaError_t e = cudaMalloc(&env->workspace, off);
  if (e != cudaSuccess) {
    delete env;
    return cuda_fail(nullptr, e, "cudaMalloc(workspace)");
  }
  env->status = reinterpret_cast<Status*>(env->workspace);
  env->w_policy_f32 = reinterpret_cast<float*>(env->workspace + pol_off);
  env->w_value_f32 = cfg->has_value ? reinterpret_cast<float*>(env->workspace + val_off) : nullptr;
  if (cfg->mlp_mode == AUV_MLP_BF16) {
    env->w_policy_packed = env->workspace + pol_pk_off;
    env->w_value_packed = env->workspace + val_pk_off;
  } else if (cfg->mlp_mode == AUV_MLP_TF32) {
    env->w_policy_packed = env->workspace + pol_pk_off;
  }
  Status s0 = {0, 0, INT_MAX, 0};
  e = cudaMemcpy(env->status, &s0, sizeof(s0), cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    cudaFree(env->workspace);
    delete env;
    return cuda_fail(nullptr, e, "init status");
  }
  *out = env;
  return AUV_OK;
}

int env_destroy(auv_env* env) {
  if (!env) return AUV_ERR_INVALID;
  cudaDeviceSynchronize();
  cudaError_t e = cudaFree(env->workspace);
  if (env->stage) cudaFree(env->stage);
  if (env->adj_scratch) cudaFree(env->adj_scratch);
  if (env->shac_ws) cudaFree(env->shac_ws);
  for (int b = 0; b < 2; ++b) {
    if (env->seg_done[b]) cudaEventDestroy(env->seg_done[b]);
    if (env->copy_done[b]) cudaEventDestroy(env->copy_done[b]);
  }
  if (env->copy_stream) cudaStreamDestroy(env->copy_stream);
  delete env;
  return e == cudaSuccess ? AUV_OK : AUV_ERR_CUDA;
}

int env_set_weights(auv_env* env, const float* policy, const float* value, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (!policy) return fail(env, AUV_ERR_INVALID, "policy weights are NULL");
  if (env->cfg.has_value && !value) return fail(env, AUV_ERR_INVALID, "value weights are NULL");
  if (!env->cfg.has_value && value)
    return fail(env, AUV_ERR_INVALID, "value weights given but has_value = 0");
  cudaError_t e = cudaMemcpyAsync(env->w_policy_f32, policy, env->policy_count * 4,
                                  cudaMemcpyDefault, s);
  if (e != cudaSuccess) return cuda_fail(env, e, "copy policy weights");
  if (value) {
    e = cudaMemcpyAsync(env->w_value_f32, value, env->value_count * 4, cudaMemcpyDefault, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "copy value weights");
  }
  if (env->cfg.mlp_mode == AUV_MLP_BF16) {
    e = auv::launch_pack_bf16(env->model, env->w_policy_f32, env->w_value_f32,
                              env->w_policy_packed, env->w_value_packed, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "pack bf16 weights");
  } else if (env->cfg.mlp_mode == AUV_MLP_TF32) {
    e = auv::launch_pack_tf32(env->model, env->w_policy_f32, env->w_policy_packed, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "pack tf32 weights");
  }
  // host sources are read before return
  void* d = nullptr;
  if (classify(policy, &d) != kDevice || (value && classify(value, &d) != kDevice)) {
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return cuda_fail(env, e, "synchronise weight upload");
  }
  env->weights_set = true;
  return AUV_OK;
}

int env_reset(auv_env* env, const uint8_t* mask, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (mask && (rc = check_device_buffer(env, mask, "mask", 1))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = is_paper(&env->cfg) ? auv::launch_paper_reset(env->model, env->buf, mask, s)
                                      : auv::launch_reset(env->model, env->buf, mask, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "reset kernel");
}

namespace {

// The kernels of T control steps from global step t_g0 (bf16 mode: the fused
// rollout, then the value network over the observations just written).
cudaError_t launch_rollout_any(auv_env* env, const Traj& tr, int T, uint64_t t_g0,
                               cudaStream_t s) {
  if (env->cfg.mlp_mode == AUV_MLP_FP32)
    return is_paper(&env->cfg)
               ? auv::launch_paper_rollout_fp32(env->model, env->buf, env->w_policy_f32,
                                                env->w_value_f32, tr, T, t_g0, env->status, s)
               : auv::launch_rollout_fp32(env->model, env->buf, env->w_policy_f32,
                                          env->w_value_f32, tr, T, t_g0, env->status, s);
  if (env->cfg.mlp_mode == AUV_MLP_TF32)
    return auv::launch_rollout_tf32(env->model, env->buf, env->w_policy_packed, tr, T, t_g0,
                                    env->status, s);
  cudaError_t e = auv::launch_rollout_bf16(env->model, env->buf, env->w_policy_packed, tr, T,
                                           t_g0, env->status, s);
  if (e != cudaSuccess || !tr.value) return e;
  return auv::launch_value_bf16(env->model, env->w_value_packed, env->w_value_f32, tr.obs,
                                (size_t)T * env->model.n, env->model.n, tr.value, env->status, s);
}

constexpr int kTrajArrays = 6;   // obs, act, logp, value, rew, done (auv_traj order)

void** traj_slot(Traj& t, int k) {
  void** p[kTrajArrays] = {reinterpret_cast<void**>(&t.obs), reinterpret_cast<void**>(&t.act),
                           reinterpret_cast<void**>(&t.logp), reinterpret_cast<void**>(&t.value),
                           reinterpret_cast<void**>(&t.rew), reinterpret_cast<void**>(&t.done)};
  return p[k];
}

// Host trajectory arrays are filled through device staging: the steps run in
// segments of `seg` steps into one of two device segment buffers, and each
// finished segment is copied to the caller's page-locked arrays on the env's
// copy stream while the next segment computes.  The caller's stream waits
// for the last copy, so its completion still means the arrays are written.
int rollout_staged(auv_env* env, int T, const auv_traj* traj, Traj mapped,
                   const bool host[kTrajArrays], cudaStream_t s) {
  const size_t n = env->model.n;
  const size_t row[kTrajArrays] = {obs_dim(&env->cfg) * n * 4, act_dim(&env->cfg) * n * 4,
                                   n * 4, n * 4, n * 4, n};
  void* const dst[kTrajArrays] = {traj->obs, traj->act, traj->logp, traj->value, traj->rew,
                                  traj->done};
  size_t step_bytes = 0;
  for (int k = 0; k < kTrajArrays; ++k)
    if (host[k]) step_bytes += row[k];
  // about 64 MiB per segment buffer: a power of two of steps in [4, T]
  int seg = 4;
  while (seg < T && (size_t)(2 * seg) * step_bytes <= ((size_t)1 << 26)) seg *= 2;
  if (seg > T) seg = T;
  size_t off[kTrajArrays], half = 0;
  for (int k = 0; k < kTrajArrays; ++k) {
    off[k] = half;
    if (host[k]) half += ((size_t)seg * row[k] + 255) & ~(size_t)255;
  }
  cudaError_t e;
  if (!env->copy_stream) {
    if ((e = cudaStreamCreateWithFlags(&env->copy_stream, cudaStreamNonBlocking)) != cudaSuccess)
      return cuda_fail(env, e, "create copy stream");
    for (int b = 0; b < 2; ++b) {
      if ((e = cudaEventCreateWithFlags(&env->seg_done[b], cudaEventDisableTiming)) != cudaSuccess ||
          (e = cudaEventCreateWithFlags(&env->copy_done[b], cudaEventDisableTiming)) != cudaSuccess)
        return cuda_fail(env, e, "create staging events");
    }
  }
  if (2 * half > env->stage_bytes) {
    if (env->stage) {   // the previous call's copies may still read the old buffers
      if ((e = cudaStreamSynchronize(env->copy_stream)) != cudaSuccess)
        return cuda_fail(env, e, "drain copy stream");
      cudaFree(env->stage);
      env->stage = nullptr;
      env->stage_bytes = 0;
      env->last_copy = -1;
    }
    if ((e = cudaMalloc(&env->stage, 2 * half)) != cudaSuccess)
      return cuda_fail(env, e, "cudaMalloc(trajectory staging)");
    env->stage_bytes = 2 * half;
  }
  // buffers are reused across calls: start after the previous call's copies
  if (env->last_copy >= 0 && (e = cudaStreamWaitEvent(s, env->copy_done[env->last_copy], 0)) != cudaSuccess)
    return cuda_fail(env, e, "order after previous copies");
  int b = 0;
  for (int t0 = 0, j = 0; t0 < T; t0 += seg, ++j) {
    const int len = T - t0 < seg ? T - t0 : seg;
    b = j & 1;
    if (j >= 2 && (e = cudaStreamWaitEvent(s, env->copy_done[b], 0)) != cudaSuccess)
      return cuda_fail(env, e, "wait for segment buffer");
    Traj ts = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
    for (int k = 0; k < kTrajArrays; ++k) {
      void* m = *traj_slot(mapped, k);
      if (!m) continue;
      *traj_slot(ts, k) = host[k] ? static_cast<void*>(env->stage + b * half + off[k])
                                  : static_cast<void*>(static_cast<char*>(m) + (size_t)t0 * row[k]);
    }
    if ((e = launch_rollout_any(env, ts, len, env->t_g + (uint64_t)t0, s)) != cudaSuccess)
      return cuda_fail(env, e, "rollout kernels");
    if ((e = cudaEventRecord(env->seg_done[b], s)) != cudaSuccess ||
        (e = cudaStreamWaitEvent(env->copy_stream, env->seg_done[b], 0)) != cudaSuccess)
      return cuda_fail(env, e, "order segment copy");
    for (int k = 0; k < kTrajArrays; ++k) {
      if (!host[k]) continue;
      e = cudaMemcpyAsync(static_cast<char*>(dst[k]) + (size_t)t0 * row[k], env->stage + b * half + off[k],
                          (size_t)len * row[k], cudaMemcpyDeviceToHost, env->copy_stream);
      if (e != cudaSuccess) return cuda_fail(env, e, "copy trajectory segment");
    }
    if ((e = cudaEventRecord(env->copy_done[b], env->copy_stream)) != cudaSuccess)
      return cuda_fail(env, e, "record segment copy");
  }
  env->last_copy = b;
  if ((e = cudaStreamWaitEvent(s, env->copy_done[b], 0)) != cudaSuccess)
    return cuda_fail(env, e, "order after last copy");
  return AUV_OK;
}

}  // namespace

int env_rollout(auv_env* env, int T, const auv_traj* traj, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1) return fail(env, AUV_ERR_INVALID, "T must be >= 1");
  if (!env->weights_set) return fail(env, AUV_ERR_INVALID, "weights not set");
  Traj tr = {nullptr, nullptr, nullptr, nullptr, nullptr, nullptr};
  bool host[kTrajArrays] = {false, false, false, false, false, false};
  bool any_host = false;
  if (traj) {
    const char* names[kTrajArrays] = {"traj.obs", "traj.act", "traj.logp", "traj.value",
                                      "traj.rew", "traj.done"};
    void* const given[kTrajArrays] = {traj->obs, traj->act, traj->logp, traj->value, traj->rew,
                                      traj->done};
    for (int k = 0; k < kTrajArrays; ++k) {
      void* d;
      if ((rc = map_output(env, given[k], names[k], k == 5 ? 1 : 4, &d))) return rc;
      *traj_slot(tr, k) = d;
      host[k] = given[k] && classify(given[k], &d) == kHostMapped;
      any_host |= host[k];
    }
  }
  if (tr.value && !env->cfg.has_value)
    return fail(env, AUV_ERR_INVALID, "traj.value requested but has_value = 0");
  if (env->cfg.mlp_mode != AUV_MLP_FP32 && tr.value && !tr.obs)
    return fail(env, AUV_ERR_INVALID, "bf16 mode computes traj.value from traj.obs: give both");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (any_host && T >= 2) {
    if ((rc = rollout_staged(env, T, traj, tr, host, s))) return rc;
  } else {
    // device arrays, or one step: host arrays are written in place (mapped)
    cudaError_t e = launch_rollout_any(env, tr, T, env->t_g, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "rollout kernels");
  }
  env->t_g += (uint64_t)T;
  return AUV_OK;
}

int env_value(auv_env* env, const float* obs, int T, float* value, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1) return fail(env, AUV_ERR_INVALID, "T must be >= 1");
  if (!env->cfg.has_value) return fail(env, AUV_ERR_INVALID, "has_value = 0");
  if (!env->weights_set) return fail(env, AUV_ERR_INVALID, "weights not set");
  void *o, *v;
  if (!obs || !value) return fail(env, AUV_ERR_INVALID, "obs and value are required");
  if ((rc = map_output(env, const_cast<float*>(obs), "obs", 4, &o))) return rc;
  if ((rc = map_output(env, value, "value", 4, &v))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t rows = (size_t)T * env->model.n;
  cudaError_t e;
  if (env->cfg.mlp_mode == AUV_MLP_TF32)
    return fail(env, AUV_ERR_UNSUPPORTED, "tf32 mode has no value network");
  if (env->cfg.mlp_mode == AUV_MLP_FP32)
    e = auv::launch_value_fp32(env->model, env->w_value_f32, static_cast<const float*>(o), rows,
                               env->model.n, static_cast<float*>(v), s);
  else
    e = auv::launch_value_bf16(env->model, env->w_value_packed, env->w_value_f32,
                               static_cast<const float*>(o), rows, env->model.n,
                               static_cast<float*>(v), env->status, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "value kernel");
}

int env_gae(auv_env* env, int T, const float* rew, const uint8_t* done, const float* value,
            const float* last_value, float gamma, float lambda, float* adv, float* ret,
            void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1) return fail(env, AUV_ERR_INVALID, "T must be >= 1");
  if (!(gamma >= 0.0f && gamma <= 1.0f) || !(lambda >= 0.0f && lambda <= 1.0f))
    return fail(env, AUV_ERR_INVALID, "gamma and lambda must lie in [0, 1]");
  if ((rc = check_device_buffer(env, rew, "rew", 4)) || (rc = check_device_buffer(env, done, "done", 1)) ||
      (rc = check_device_buffer(env, value, "value", 4)) ||
      (rc = check_device_buffer(env, last_value, "last_value", 4)) ||
      (rc = check_device_buffer(env, adv, "adv", 4)) || (rc = check_device_buffer(env, ret, "ret", 4)))
    return rc;
  const size_t bytes = (size_t)T * env->model.n * 4;
  auto overlap = [](const void* a, size_t na, const void* b, size_t nb) {
    const char *pa = static_cast<const char*>(a), *pb = static_cast<const char*>(b);
    return pa < pb + nb && pb < pa + na;
  };
  const size_t nd = (size_t)T * env->model.n, nl = (size_t)env->model.n * 4;
  for (const void* out : {static_cast<const void*>(adv), static_cast<const void*>(ret)})
    if (overlap(out, bytes, rew, bytes) || overlap(out, bytes, value, bytes) ||
        overlap(out, bytes, done, nd) || overlap(out, bytes, last_value, nl))
      return fail(env, AUV_ERR_INVALID, "adv and ret must not overlap the inputs");
  if (overlap(adv, bytes, ret, bytes)) return fail(env, AUV_ERR_INVALID, "adv overlaps ret");
  cudaError_t e = auv::launch_gae(env->model.n, T, rew, done, value, last_value, gamma, lambda,
                                  adv, ret, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "gae kernel");
}

int env_step(auv_env* env, float* obs_out, float* rew_out, uint8_t* done_out, void* stream) {
  auv_traj tr = {obs_out, nullptr, nullptr, nullptr, rew_out, done_out};
  return env_rollout(env, 1, &tr, stream);
}

int env_step_actions(auv_env* env, const float* act, int T, float* rew_out, uint8_t* done_out,
                     float* state_trace, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1) return fail(env, AUV_ERR_INVALID, "T must be >= 1");
  if ((rc = check_device_buffer(env, act, "act", 4))) return rc;
  void *rew, *done, *trace;
  if (!rew_out || !done_out) return fail(env, AUV_ERR_INVALID, "rew_out and done_out are required");
  if ((rc = map_output(env, rew_out, "rew_out", 4, &rew))) return rc;
  if ((rc = map_output(env, done_out, "done_out", 1, &done))) return rc;
  if ((rc = map_output(env, state_trace, "state_trace", 4, &trace))) return rc;
  cudaError_t e = is_paper(&env->cfg)
      ? auv::launch_paper_replay(env->model, env->buf, act, T, static_cast<float*>(rew),
                                 static_cast<uint8_t*>(done), static_cast<float*>(trace),
                                 env->status, static_cast<cudaStream_t>(stream))
      : auv::launch_replay(env->model, env->buf, act, T, static_cast<float*>(rew),
                                     static_cast<uint8_t*>(done), static_cast<float*>(trace),
                                     env->status, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "replay kernel");
}

int env_adjoint(auv_env* env, int T, const float* act, const float* coef, const float* lam_T,
                float* grad_act, float* lam_0, float* rew_out, uint8_t* done_out, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1 || T > AUV_ADJOINT_MAX_T)
    return fail(env, AUV_ERR_INVALID, "T outside [1, %d]", AUV_ADJOINT_MAX_T);
  if (env->model.substeps > AUV_ADJOINT_MAX_SUBSTEPS)
    return fail(env, AUV_ERR_UNSUPPORTED, "the adjoint supports at most %d substeps",
                AUV_ADJOINT_MAX_SUBSTEPS);
  if ((rc = check_device_buffer(env, act, "act", 4)) || (rc = check_device_buffer(env, coef, "coef", 4)) ||
      (rc = check_device_buffer(env, grad_act, "grad_act", 4)))
    return rc;
  if (lam_T && (rc = check_device_buffer(env, lam_T, "lam_T", 4))) return rc;
  void *l0 = nullptr, *rew = nullptr, *done = nullptr;
  if ((rc = map_output(env, lam_0, "lam_0", 4, &l0)) || (rc = map_output(env, rew_out, "rew_out", 4, &rew)) ||
      (rc = map_output(env, done_out, "done_out", 1, &done)))
    return rc;
  const size_t need = auv::adjoint_scratch_floats(env->model.n, T);
  if (need > env->adj_scratch_floats) {
    if (env->adj_scratch) {
      cudaError_t e = cudaFree(env->adj_scratch);
      env->adj_scratch = nullptr;
      env->adj_scratch_floats = 0;
      if (e != cudaSuccess) return cuda_fail(env, e, "free adjoint scratch");
    }
    cudaError_t e = cudaMalloc(&env->adj_scratch, need * sizeof(float));
    if (e != cudaSuccess) {
      env->adj_scratch = nullptr;
      return cuda_fail(env, e, "cudaMalloc(adjoint scratch)");
    }
    env->adj_scratch_floats = need;
  }
  cudaError_t e = auv::launch_adjoint(env->model, env->buf, act, T, coef, lam_T, grad_act,
                                      static_cast<float*>(l0), static_cast<float*>(rew),
                                      static_cast<uint8_t*>(done), env->adj_scratch, env->status,
                                      static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "adjoint kernel");
}

int env_shac_window(auv_env* env, const float* policy, const float* value, int T,
                    const float* coef, float coef_V, uint32_t precision, float* grad,
                    float* J_out, float* obs_out, float* rew_out, uint8_t* done_out,
                    void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (T < 1 || T > AUV_ADJOINT_MAX_T)
    return fail(env, AUV_ERR_INVALID, "T outside [1, %d]", AUV_ADJOINT_MAX_T);
  if (env->model.substeps > AUV_ADJOINT_MAX_SUBSTEPS)
    return fail(env, AUV_ERR_UNSUPPORTED, "the SHAC window supports at most %d substeps",
                AUV_ADJOINT_MAX_SUBSTEPS);
  const int H = (int)env->cfg.hidden;
  if (H < 8 || H > 1024 || H % 8)
    return fail(env, AUV_ERR_UNSUPPORTED, "the SHAC window needs hidden a multiple of 8 in [8, 1024]");
  if (!std::isfinite(coef_V)) return fail(env, AUV_ERR_INVALID, "coef_V not finite");
  if (precision != AUV_PPO_FP32 && precision != AUV_PPO_TF32)
    return fail(env, AUV_ERR_INVALID, "precision must be AUV_PPO_FP32 or AUV_PPO_TF32");
  if ((rc = check_device_buffer(env, policy, "policy", 4)) ||
      (rc = check_device_buffer(env, coef, "coef", 4)) ||
      (rc = check_device_buffer(env, grad, "grad", 4)))
    return rc;
  if (value && (rc = check_device_buffer(env, value, "value", 4))) return rc;
  if (obs_out && (rc = check_device_buffer(env, obs_out, "obs_out", 4))) return rc;
  void *J = nullptr, *rew = nullptr, *done = nullptr;
  if ((rc = map_output(env, J_out, "J_out", 4, &J)) ||
      (rc = map_output(env, rew_out, "rew_out", 4, &rew)) ||
      (rc = map_output(env, done_out, "done_out", 1, &done)))
    return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const auv::shac::Layout L = auv::shac::layout(env->model.n, T, H, is_paper(&env->cfg));
  if (L.bytes > env->shac_ws_bytes || T != env->shac_T) {
    if (L.bytes > env->shac_ws_bytes) {
      if (env->shac_ws) {
        cudaError_t e = cudaFree(env->shac_ws);
        env->shac_ws = nullptr;
        env->shac_ws_bytes = 0;
        if (e != cudaSuccess) return cuda_fail(env, e, "free SHAC workspace");
      }
      cudaError_t e = cudaMalloc(&env->shac_ws, L.bytes);
      if (e != cudaSuccess) {
        env->shac_ws = nullptr;
        return cuda_fail(env, e, "cudaMalloc(SHAC workspace)");
      }
      env->shac_ws_bytes = L.bytes;
    }
    cudaError_t e = auv::shac::init(L, env->shac_ws, s);
    if (e != cudaSuccess) return cuda_fail(env, e, "initialise SHAC workspace");
    env->shac_T = T;
  }
  rc = auv::shac::run_window(env->model, env->buf, env->status, L, env->shac_ws,
                             env->t_g, policy, value, coef, coef_V, precision == AUV_PPO_TF32,
                             grad, static_cast<float*>(J),
                             obs_out, static_cast<float*>(rew), static_cast<uint8_t*>(done), s,
                             env->err);
  if (rc != AUV_OK) return rc;
  env->t_g += (uint64_t)T;
  return AUV_OK;
}

int env_inverse_allocate(auv_env* env, int n, const float* wrench, float* cmd, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (n < 1) return fail(env, AUV_ERR_INVALID, "n must be >= 1");
  if ((rc = check_device_buffer(env, wrench, "wrench", 4))) return rc;
  void* out = nullptr;
  if (!cmd) return fail(env, AUV_ERR_INVALID, "cmd is NULL");
  if ((rc = map_output(env, cmd, "cmd", 4, &out))) return rc;
  if (!env->inv_ready) {
    if (!auv::pinv_6x8(env->model.alloc_t, env->inv.pinv))
      return fail(env, AUV_ERR_UNSUPPORTED, "the allocation matrix has rank < 6");
    env->inv_ready = true;
  }
  cudaError_t e = auv::launch_inverse_alloc(n, env->inv, wrench, static_cast<float*>(out),
                                            static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "inverse allocation kernel");
}

int env_observe(auv_env* env, float* obs_out, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  void* d;
  if (!obs_out) return fail(env, AUV_ERR_INVALID, "obs_out is NULL");
  if ((rc = map_output(env, obs_out, "obs_out", 4, &d))) return rc;
  cudaError_t e = is_paper(&env->cfg)
      ? auv::launch_paper_observe(env->model, env->buf, static_cast<float*>(d),
                                  static_cast<cudaStream_t>(stream))
      : auv::launch_observe(env->model, env->buf, static_cast<float*>(d),
                                      static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "observe kernel");
}

int env_policy_forward(auv_env* env, const float* obs, int n, float* head, float* value,
                       void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (n < 1) return fail(env, AUV_ERR_INVALID, "n must be >= 1");
  if (!env->weights_set) return fail(env, AUV_ERR_INVALID, "weights not set");
  if ((rc = check_device_buffer(env, obs, "obs", 4))) return rc;
  if ((rc = check_device_buffer(env, head, "head", 4))) return rc;
  if (value && !env->cfg.has_value) return fail(env, AUV_ERR_INVALID, "value but has_value = 0");
  if (value && (rc = check_device_buffer(env, value, "value", 4))) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (env->cfg.mlp_mode == AUV_MLP_TF32)
    return fail(env, AUV_ERR_UNSUPPORTED, "tf32 mode evaluates the policy inside env_rollout only");
  if (env->cfg.mlp_mode == AUV_MLP_FP32)
    e = auv::launch_forward_fp32(env->model, env->w_policy_f32, env->w_value_f32, obs, n, head,
                                 value, s);
  else
    e = auv::launch_forward_bf16(env->model, env->w_policy_packed, env->w_value_packed,
                                 env->w_value_f32, obs, n, head, value, env->status, s);
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "forward kernel");
}

int env_draw_words(auv_env* env, uint32_t stream_id, uint64_t index, int n_blocks, uint32_t* out,
                   void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (n_blocks < 1 || n_blocks > 64) return fail(env, AUV_ERR_INVALID, "n_blocks outside [1, 64]");
  if ((rc = check_device_buffer(env, out, "out", 4))) return rc;
  cudaError_t e = auv::launch_draw_words(env->model, stream_id, index, n_blocks, out,
                                         static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "draw-words kernel");
}

int env_get_step(const auv_env* env, uint64_t* t_g) {
  if (!env || !t_g) return AUV_ERR_INVALID;
  *t_g = env->t_g;
  return AUV_OK;
}

int env_set_step(auv_env* env, uint64_t t_g) {
  if (!env) return AUV_ERR_INVALID;
  env->t_g = t_g;
  return AUV_OK;
}

int env_get_state(auv_env* env, auv_snapshot* snap, void* stream) {
  int rc = snapshot_arrays(env, snap, false);
  if (rc) return rc;
  if ((rc = check_device(env))) return rc;
  auv_layout lay;
  env_layout(env->cfg.model, &lay);
  snap->model = env->cfg.model;
  snap->n_envs = env->cfg.n_envs;
  snap->state_fields = lay.state_fields;
  snap->param_fields = lay.param_fields;
  snap->reserved = 0;
  snap->t_g = env->t_g;
  void* const dst[4] = {snap->state, snap->params, snap->t_ep, snap->episode};
  const void* const src[4] = {env->buf.state, env->buf.params, env->buf.t_ep, env->buf.episode};
  return copy_batch(env, dst, src, static_cast<cudaStream_t>(stream));
}

int env_set_state(auv_env* env, const auv_snapshot* snap, void* stream) {
  int rc = snapshot_arrays(env, snap, true);
  if (rc) return rc;
  if ((rc = check_device(env))) return rc;
  void* const dst[4] = {env->buf.state, env->buf.params, env->buf.t_ep, env->buf.episode};
  const void* const src[4] = {snap->state, snap->params, snap->t_ep, snap->episode};
  rc = copy_batch(env, dst, src, static_cast<cudaStream_t>(stream));
  if (rc) return rc;
  env->t_g = snap->t_g;
  return AUV_OK;
}

int env_status(auv_env* env, auv_status* out, void* stream) {
  if (!env || !out) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(env, e, "synchronise");
  Status st;
  e = cudaMemcpy(&st, env->status, sizeof(st), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(env, e, "read status");
  out->code = st.code;
  out->nan_flag = st.nan_flag;
  out->first_nan_env = st.first_nan_env == INT_MAX ? -1 : st.first_nan_env;
  out->timeouts = st.timeouts;
  if (st.code != 0)
    fail(env, st.code, "device status %d (nan_flag %d, first env %d, timeouts %d)", st.code,
         st.nan_flag, out->first_nan_env, st.timeouts);
  return st.code;
}

int env_selftest_wait_timeout(auv_env* env, uint32_t limit_us, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  if (limit_us < 1 || limit_us > 5000000)
    return fail(env, AUV_ERR_INVALID, "limit_us outside [1, 5e6]");
  cudaError_t e = auv::launch_wait_selftest(env->status, (uint64_t)limit_us * 1000ull,
                                            static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "wait self-test kernel");
}

int env_clear_status(auv_env* env, void* stream) {
  if (!env) return AUV_ERR_INVALID;
  int rc = check_device(env);
  if (rc) return rc;
  static const Status s0 = {0, 0, INT_MAX, 0};
  cudaError_t e = cudaMemcpyAsync(env->status, &s0, sizeof(s0), cudaMemcpyHostToDevice,
                                  static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? AUV_OK : cuda_fail(env, e, "clear status");
}

}  // extern "C"
