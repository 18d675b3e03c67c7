/*
 * auvenv.h -- C ABI of the GB300 batched AUV rollout library (libauvenv.so).
 *
 * The library steps N independent underwater-vehicle environments of the
 * 6-DOF position-control task of "Fast Policy Learning for 6-DOF Position
 * Control of Underwater Vehicles" (arXiv 2512.13359): per control step it
 * evaluates the policy network on each env's observation, samples a Gaussian
 * action, maps it through the thruster allocation to a body wrench,
 * integrates the rigid-body + hydrodynamic model, and computes the reward,
 * the done flag and the automatic reset (paper §IV-A: batched simulation of
 * independent environments sharing one model and integrator).
 *
 * Two environment models (auv_config.model):
 *  - AUV_MODEL_FOSSEN: the thruster-level model -- Fossen's 6-DOF equations
 *    with added mass, Coriolis, linear + quadratic damping, restoring forces,
 *    a water current and per-env randomised parameters; 8 thruster commands
 *    through an allocation matrix; 18-float observation.
 *  - AUV_MODEL_PAPER: the paper's own environment (§IV-B): a normalised body
 *    wrench scaled by F_max and tau_max (Eq. 1); a free rigid body under the
 *    inertia-box fluid model (quadratic drag and viscous resistance of the
 *    uniform box with the body's mass and inertia); buoyancy folded into an
 *    effective gravity randomised per episode (§IV-C); a 12-float
 *    observation with the axis-angle attitude error (§IV-B1); the five-term
 *    reward of Eqs. (2)-(7).
 * The sizes that differ between the models are given by env_layout().
 *
 * Conventions shared by every entry point
 *  - Return value: AUV_OK (0) or a negative AUV_ERR_* code; env_last_error()
 *    gives a one-line reason.  No entry point aborts or traps.
 *  - Asynchrony: every call that takes `stream` (a cudaStream_t; NULL = the
 *    legacy default stream) only enqueues work on that stream and returns.
 *    Device-side faults (non-finite state, a wait that timed out) are latched
 *    in a device status block and reported by env_status().
 *  - Layout: all per-env arrays are structure-of-arrays, env index fastest:
 *    element (k, i) of a [K][N] array is at k*N + i; trajectory arrays are
 *    [T][K][N] with element (t, k, i) at (t*K + k)*N + i.
 *  - Ownership: the caller allocates and owns every state, parameter and
 *    trajectory buffer (device memory, or host memory that is page-locked and
 *    mapped, e.g. from cudaHostAlloc, for trajectory outputs).  The library
 *    owns only its handle and a device workspace it allocates in env_create
 *    and frees in env_destroy (packed network weights and the status block).
 *  - The CUDA device is the one current on the calling thread at env_create;
 *    later calls must be made with the same device current.
 */
#ifndef AUVENV_H
#define AUVENV_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define AUV_ABI_VERSION 3

/* status codes */
#define AUV_OK 0
#define AUV_ERR_INVALID (-1)      /* bad argument or configuration value     */
#define AUV_ERR_SIZE (-2)         /* buffer missing, misaligned or wrong kind */
#define AUV_ERR_CUDA (-3)         /* a CUDA runtime call failed              */
#define AUV_ERR_TIMEOUT (-4)      /* a device-side bounded wait gave up      */
#define AUV_ERR_NAN (-5)          /* non-finite state detected               */
#define AUV_ERR_UNSUPPORTED (-6)  /* valid but not implemented combination   */

/* network arithmetic */
#define AUV_MLP_FP32 0   /* fp32 operands and accumulation on CUDA cores        */
#define AUV_MLP_BF16 1   /* bf16 weights/activations, fp32 accumulation, tcgen05 */
#define AUV_MLP_TF32 2   /* fp32 networks with tf32 operands (rounded to nearest),
                            fp32 accumulation, tcgen05 kind::tf32: Fossen model,
                            hidden 256, policy_out 8 or 16, no value network;
                            env_rollout only (env_value and env_policy_forward
                            return AUV_ERR_UNSUPPORTED) */

/* environment models */
#define AUV_MODEL_FOSSEN 0
#define AUV_MODEL_PAPER 1

/* sizes fixed by the Fossen model */
#define AUV_OBS_DIM 18      /* observation: dp_b(3), R_e column-major(9), v(3), w(3) */
#define AUV_ACT_DIM 8       /* normalised thruster commands                        */
#define AUV_STATE_FIELDS 19 /* p(3) q(4: w,x,y,z body->world) nu(6) nu_prev(6)     */
#define AUV_PARAM_FIELDS 17 /* p_d(3) q_d(4) s_m s_a s_d dB r_b(3) V_c(3)          */

/* sizes fixed by the paper model */
#define AUV_PAPER_OBS_DIM 12      /* dp_b(3), axis-angle error(3), v(3), w(3)        */
#define AUV_PAPER_ACT_DIM 6       /* normalised wrench F(3), tau(3)                  */
#define AUV_PAPER_HIST 8          /* action-history slots kept (mavg_len <= 8)       */
#define AUV_PAPER_STATE_FIELDS 61 /* p(3) q(4) nu(6) history[8][6] of clipped actions */
#define AUV_PAPER_PARAM_FIELDS 8  /* p_d(3) q_d(4) g_eff                             */

/*
 * Model and workload description.  Paper §IV-B (environment), §IV-C (domain
 * randomisation), §IV-D (Fossen 6-DOF equations of motion), Eqs. (1)-(7)
 * (action and reward), §V-A1 (episodes with a random reference).
 * The equations of motion, in the body frame, with nu = [v; w]:
 *   (M_RB + M_A) nu' = tau - C_RB(nu) nu - C_A(nu_r) nu_r - D(nu_r) nu_r
 *                      - g(eta) + M_A nu_c'
 * nu_r = nu - [R^T V_c; 0], M_RB = diag(m, m, m, I), M_A, D_L, D_Q diagonal,
 * damping D(nu_r) nu_r = (D_L + D_Q |nu_r|) nu_r, weight at the origin,
 * buoyancy B = m |g| + dB at r_b, tau = alloc * (thrust_max * clip(a, -1, 1)).
 * Per episode the randomised scales multiply: s_m the mass and inertia, s_a
 * the added mass, s_d both damping matrices.
 */
typedef struct auv_config {
  uint32_t struct_size;   /* sizeof(auv_config): version guard               */
  uint32_t n_envs;        /* N >= 1                                          */
  uint32_t substeps;      /* physics substeps per control step, 1..64        */
  uint32_t episode_len;   /* control steps per episode (time-limit done) >= 1 */
  uint32_t seed;          /* Philox key word 1 (word 0 is the env id)        */
  uint32_t env_id_base;   /* global id of local env 0: env i uses Philox key
                             word 0 = env_id_base + i, so a shard of a larger
                             batch reproduces that batch's envs exactly       */
  uint32_t dr_enable;     /* 1: draw s_m, s_a, s_d, dB, r_b at every reset   */
  float dt;               /* control period [s] > 0                          */
  float mass;             /* m [kg]                                          */
  float inertia[3];       /* principal moments about the CoG [kg m^2]        */
  float added_mass[6];    /* diag(M_A)                                       */
  float damp_lin[6];      /* diag(D_L)                                       */
  float damp_quad[6];     /* diag(D_Q)                                       */
  float gravity[3];       /* world gravity vector g_w [m/s^2]                */
  float thrust_max;       /* newtons per thruster at |a| = 1                 */
  float alloc[48];        /* allocation matrix, row-major [6][8]             */
  float w_pos, w_att, w_act, w_vs;  /* reward weights (see env_rollout)      */
  float init_pos_range;   /* initial position U[-r, r] per axis [m]          */
  float init_att_range;   /* initial roll, pitch, yaw U[-r, r] [rad]         */
  float goal_pos_range;   /* goal position U[-r, r] per axis [m]             */
  float goal_yaw_range;   /* goal yaw U[-r, r] [rad], r <= pi                */
  float current_range;    /* water current U[-r, r] per world axis [m/s]     */
  float dr_scale_lo, dr_scale_hi;   /* s_m, s_a, s_d ~ U[lo, hi]             */
  float dr_buoy_range;    /* dB ~ U[-r, r] [N]                               */
  float dr_cob_range;     /* r_b ~ U[-r, r] per axis [m]                     */
  uint32_t hidden;        /* hidden width H of both networks                 */
  uint32_t policy_out;    /* 8: mean only (fixed log-std); 16: mean + log-std */
  uint32_t mlp_mode;      /* AUV_MLP_FP32, AUV_MLP_BF16 or AUV_MLP_TF32      */
  uint32_t has_value;     /* 1: value network present                        */
  float logstd_fixed[8];  /* log-std used when policy_out == 8               */
  float logstd_min, logstd_max;     /* clamp of the log-std head             */
  /* ---- model selection and the paper model (AUV_MODEL_PAPER) ----------- *
   * The paper model uses n_envs, substeps, episode_len, seed, env_id_base,  *
   * dr_enable, dt, mass, inertia, w_pos, w_att, w_act, init_pos_range,      *
   * init_att_range, goal_pos_range, the network fields (policy_out 6: mean  *
   * with logstd_fixed[0..5], or 12: mean + log-std head) and the fields     *
   * below; it ignores the Fossen-only fields.                               */
  uint32_t model;         /* AUV_MODEL_FOSSEN or AUV_MODEL_PAPER             */
  float f_max, tau_max;   /* Eq. (1): force [N] and torque [N m] at |a| = 1  */
  float fluid_density;    /* rho [kg/m^3] of the inertia-box fluid model     */
  float fluid_viscosity;  /* mu [Pa s]                                       */
  float g_eff;            /* nominal effective gravity along world -z [m/s^2] */
  float dr_gravity_range; /* g_eff + U[-r, r] at every reset if dr_enable    */
  float goal_att_range;   /* goal roll, pitch, yaw U[-r, r] [rad], r <= pi   */
  float w_axes[3];        /* D = diag(w_x, w_y, w_z) of Eq. (3)              */
  float w_vel, w_mavg;    /* Eq. (6) and Eq. (7) weights                     */
  uint32_t mavg_len;      /* K: previous actions averaged in Eq. (7), 1..8   */
} auv_config;

/* Sizes of one model's arrays (see env_layout). */
typedef struct auv_layout {
  uint32_t obs_dim;       /* rows of an observation                          */
  uint32_t act_dim;       /* rows of an action                               */
  uint32_t state_fields;  /* rows of auv_buffers.state                       */
  uint32_t param_fields;  /* rows of auv_buffers.params                      */
} auv_layout;

/* Caller-owned device buffers holding the batch (SoA, see layout above);
 * row counts for the paper model from env_layout. */
typedef struct auv_buffers {
  float* state;       /* [19][N] p, q, nu, nu_prev                       */
  float* params;      /* [17][N] p_d, q_d, s_m, s_a, s_d, dB, r_b, V_c    */
  int32_t* t_ep;      /* [N] control steps taken in the current episode  */
  uint32_t* episode;  /* [N] index of the next episode's reset draw      */
} auv_buffers;

/* Trajectory outputs of env_rollout; any pointer may be NULL (not written).
 * The row counts 18 and 8 below are the Fossen model's obs_dim and act_dim;
 * the paper model writes obs[T][12][N] and act[T][6][N].
 * Device memory or mapped page-locked host memory, 4-byte aligned (done:
 * any alignment).  Host arrays are filled through device staging buffers
 * (see env_rollout).                                                      */
typedef struct auv_traj {
  float* obs;     /* [T][18][N] observation the action was taken from   */
  float* act;     /* [T][8][N]  unclipped sampled action a_t            */
  float* logp;    /* [T][N]     log pi(a_t | o_t)                       */
  float* value;   /* [T][N]     V(o_t) (needs has_value)                */
  float* rew;     /* [T][N]     reward r_t on the post-step state       */
  uint8_t* done;  /* [T][N]     1 if the episode ended at this step     */
} auv_traj;

/* Device status block contents, read by env_status(). */
typedef struct auv_status {
  int32_t code;          /* AUV_OK, AUV_ERR_NAN or AUV_ERR_TIMEOUT (first latched) */
  int32_t nan_flag;      /* 1 if any env produced a non-finite state               */
  int32_t first_nan_env; /* smallest env id with a non-finite state, or -1         */
  int32_t timeouts;      /* number of device waits that gave up                    */
} auv_status;

typedef struct auv_env auv_env;

/* ABI version of the loaded library (AUV_ABI_VERSION it was built with). */
int env_abi_version(void);

/* env_layout: array sizes of environment model `model` (AUV_MODEL_*);
 * AUV_ERR_INVALID for an unknown model. */
int env_layout(uint32_t model, auv_layout* out);

/*
 * env_create: validate `cfg`, bind the caller's buffers and allocate the
 * library workspace on the current device.  Writes the handle to *out.
 * Buffers must hold N elements per field and be 16-byte aligned.  Nothing is
 * initialised: call env_set_weights and env_reset before stepping.  The
 * global step counter (the action-noise stream index) starts at 0.
 * Errors: AUV_ERR_INVALID (bad cfg value, NULL pointer, struct_size
 * mismatch), AUV_ERR_UNSUPPORTED (hidden/policy_out/mode combination not
 * built), AUV_ERR_CUDA.
 */
int env_create(const auv_config* cfg, const auv_buffers* buf, auv_env** out);

/* env_destroy: synchronise the device, free the workspace and the handle. */
int env_destroy(auv_env* env);

/* One-line description of the last error on this handle ("" if none). */
const char* env_last_error(const auv_env* env);

/*
 * env_set_weights: load the policy (and value) network weights.  Layout per
 * network, fp32, row-major [out][in]: W1[H][18] b1[H] W2[H][H] b2[H]
 * W3[O][H] b3[O] with O = policy_out (policy) or 1 (value).  Pointers may be
 * host or device memory; `value` must be non-NULL iff has_value.  The library
 * converts them into its packed device layout (bf16 rounding to nearest even
 * in AUV_MLP_BF16 mode) on `stream`; host memory is read before return.
 */
int env_set_weights(auv_env* env, const float* policy, const float* value, void* stream);

/*
 * env_reset: start a new episode for every env with mask[i] != 0 (all envs if
 * mask is NULL; mask is device memory, [N] bytes).  Draws, from Philox4x32-10
 * with key (env_id_base + i, seed) and counter (episode, 0, 1, 0..4), 20 uniforms:
 * initial position, roll/pitch/yaw, goal position, goal yaw, current, s_m,
 * s_a, s_d, dB, r_b (paper §IV-C, §V-A1); zero velocities; t_ep = 0;
 * episode += 1.  Bit-exact across implementations of the same steps.
 * Paper model: 13 uniforms (counter blocks 0..3): goal position, goal roll,
 * pitch, yaw, effective-gravity offset, initial position, initial roll,
 * pitch, yaw; velocities and the action history zero.
 */
int env_reset(auv_env* env, const uint8_t* mask, void* stream);

/*
 * env_rollout: T >= 1 control steps of the full hot path for all envs, state
 * carried on chip.  Per step t and env: o_t = observation (paper §IV-B1,
 * attitude as the rotation-matrix error of §V-A3); (mu, log sigma) = policy
 * network; eps = 8 Box-Muller normals from Philox key (env id, seed), counter
 * (t_g lo, t_g hi, 0, 0..1); a = mu + sigma eps; log pi = sum(-eps^2/2 -
 * log sigma - log(2 pi)/2); tau = alloc (thrust_max clip(a, -1, 1)) (Eq. 1 and
 * the thruster allocation of §V-B); nu_prev = nu; `substeps` semi-implicit
 * Euler substeps of the equations of motion; r = -w_pos |p - p_d| - w_att
 * theta_e - w_act |clip(a)|^2 - w_vs |nu - nu_prev|^2 (weighted norms of
 * Eqs. 2-7); t_ep += 1; done = (t_ep == episode_len); on done the env resets
 * as in env_reset.  The global step t_g advances by T.
 * Paper model: o_t is [dp_b, axis-angle error of conj(q_d) (x) q, v, w]; a
 * takes the first 6 of the 8 normals; a_c = clip(a, -1, 1); tau = [F_max
 * a_c(0:3); tau_max a_c(3:6)] (Eq. 1); the substeps integrate M_RB nu' = tau +
 * fluid wrench - C_RB(nu) nu + R^T (0, 0, -m g_eff); r = -w_pos |D dp_b|^2 -
 * w_att |theta_e|^2 - w_act |a_c(3:6)|^2 - w_vel |w|^2 - w_mavg |a_c - mean
 * of the previous mavg_len a_c|^2 (Eqs. 2-7, history zero after a reset),
 * then a_c enters history slot (t_ep mod mavg_len).
 * In AUV_MLP_BF16 mode traj.value (if given) comes from a value-network pass
 * over traj.obs after the steps, so traj.obs is required with it.
 * Host arrays (T >= 2): the steps run in segments into two device staging
 * buffers (allocated on the first such call, about 2 x 64 MiB, kept until
 * env_destroy); each finished segment is copied to the host arrays on a
 * copy stream of the env while the next segment computes.  `stream` waits
 * for the last copy, so its completion still means every array is written.
 * With T = 1 host arrays are written in place through their device mapping.
 * Results do not depend on where the arrays live.
 */
int env_rollout(auv_env* env, int T, const auv_traj* traj, void* stream);

/* env_step: env_rollout with T = 1 writing only obs (the observation the
 * step acted on), rew and done; each may be NULL. */
int env_step(auv_env* env, float* obs_out, float* rew_out, uint8_t* done_out, void* stream);

/*
 * env_step_actions: action replay.  T control steps with the given
 * normalised actions act[T][act_dim][N] (device) instead of the policy:
 * allocation (paper model: the Eq. (1) wrench), substeps, reward, done and
 * auto-reset exactly as in env_rollout.  Writes rew[T][N], done[T][N] and,
 * if non-NULL, state_trace[T][state_fields][N] (state after each step, after
 * any reset).  Does not advance t_g.
 */
int env_step_actions(auv_env* env, const float* act, int T, float* rew_out, uint8_t* done_out,
                     float* state_trace, void* stream);

/*
 * env_value: the value network on stored observations, in the trajectory
 * layout: obs[T][obs_dim][N] -> value[T][N] (device or mapped host memory),
 * T >= 1, with the loaded value weights (needs has_value).  A PPO learner
 * re-evaluates values this way; env_rollout calls it itself when given
 * traj.value.
 */
int env_value(auv_env* env, const float* obs, int T, float* value, void* stream);

/* env_observe: observation of the current state, obs[obs_dim][N] (device). */
int env_observe(auv_env* env, float* obs_out, void* stream);

/*
 * env_policy_forward: evaluate the loaded networks on caller observations
 * obs[n][obs_dim] (row-major, device) for n >= 1 rows: head[n][policy_out] (raw
 * outputs: mean, then unclamped log-std) and, if value is non-NULL and
 * has_value, value[n].  Same device arithmetic as env_rollout.
 */
int env_policy_forward(auv_env* env, const float* obs, int n, float* head, float* value,
                       void* stream);

/*
 * env_draw_words: the raw Philox4x32-10 words of one stream for every env:
 * out[4*n_blocks][N] (device, uint32) with block b of env i = Philox(key =
 * (env_id_base + i, seed), counter = (index lo, index hi, stream_id, b)).  stream_id 0 =
 * action noise (index = global step), 1 = reset (index = episode).
 */
int env_draw_words(auv_env* env, uint32_t stream_id, uint64_t index, int n_blocks,
                   uint32_t* out, void* stream);

/*
 * env_policy_forward_noalloc: the same network evaluation as
 * env_policy_forward in AUV_MLP_BF16 mode, for callers that must not allocate
 * device memory, e.g. an on-vehicle control loop with a hard period (an
 * allocation can synchronise the device) or a host application that owns a
 * fixed device-memory budget.  The paper has no counterpart; this is a
 * library convenience.
 *  - No handle and no allocation: the packed weights and a status word live
 *    in one static device array of 312.25 KiB that every GPU loading this
 *    library holds until the process exits.
 *  - The first call on a device is a warm-up: it looks up that array's
 *    address (once per device), and under the CUDA runtime's lazy module
 *    loading (the default) it is also the call that loads the array's module
 *    and the kernels, which may take device memory and synchronise.  Make
 *    it before the period in which nothing may allocate, and before any
 *    stream capture; later calls allocate nothing.
 *  - hidden must be 256 and policy_out 16 (the built tensor-core shape);
 *    larger values return AUV_ERR_SIZE (the packed weights would not fit
 *    the array), other values AUV_ERR_UNSUPPORTED.
 *  - policy[, value_w]: fp32 weights in the env_set_weights layout; obs[n][18]
 *    (row-major); outputs head[n][policy_out] and, iff value_w is given,
 *    value[n].  All device memory of the current device, 16-byte aligned;
 *    n >= 1.  Pointers to another GPU's memory return AUV_ERR_SIZE.
 *  - status_out (device memory of the current device, or NULL): receives the
 *    call's status block (code AUV_ERR_TIMEOUT and timeouts > 0 if a device
 *    wait gave up), copied on `stream` after the kernels.
 *  - Every call on a device shares the array and leaves its contents there:
 *    calls that overlap on the GPU (other streams, other host threads) race
 *    on it and must be serialised by the caller.
 */
int env_policy_forward_noalloc(int hidden, int policy_out, const float* policy,
                               const float* value_w, const float* obs, int n, float* head,
                               float* value, auv_status* status_out, void* stream);

/*
 * env_gae: generalised advantage estimation over a rollout's trajectory --
 * the advantage estimator of the PPO learner (paper §III-A; Schulman et al.
 * 2016).  For t = T-1 .. 0 and every env:
 *   delta_t = rew_t + gamma (1 - done_t) V_{t+1} - V_t,   V_T = last_value
 *   adv_t   = delta_t + gamma lambda (1 - done_t) adv_{t+1},  adv_T = 0
 *   ret_t   = adv_t + V_t   (the value target)
 * A done step ends its episode: nothing of the next episode flows back.
 * rew, value, adv, ret: [T][N] fp32; done: [T][N] u8; last_value: [N] (the
 * value of the observation after the last step, e.g. env_observe then
 * env_value).  All device memory, 4-byte aligned; adv and ret must not
 * overlap the inputs.  T >= 1, 0 <= gamma, lambda <= 1.
 */
int env_gae(auv_env* env, int T, const float* rew, const uint8_t* done, const float* value,
            const float* last_value, float gamma, float lambda, float* adv, float* ret,
            void* stream);

/* ---------------------------------------------------------------------------
 * PPO learner (paper §III-A: PPO with its clipped surrogate objective,
 * Schulman et al. 2017) -- the update that consumes the rollout's trajectory.
 *
 * The learner owns fp32 master weights of the two networks the rollout runs
 * (policy obs -> H -> H -> 2A: mean and log-std; value obs -> H -> H -> 1;
 * tanh hidden layers), their Adam moments and its counters.  One gradient
 * step on a minibatch of B samples computes, in float arithmetic:
 *   mu, ls = policy head (ls clamped to [logstd_min, logstd_max])
 *   logp   = sum_k -((a_k - mu_k) / e^ls_k)^2 / 2 - ls_k - log(2 pi) / 2
 *   r      = exp(logp - logp_old)
 *   A_n    = (adv - mean adv) / (std adv + 1e-8) over the minibatch (std with
 *            B - 1 in the denominator; norm_adv = 0 uses adv as is)
 *   L      = mean max(-A_n r, -A_n clip(r, 1 - clip_eps, 1 + clip_eps))
 *          + vf_coef mean (V - ret)^2 / 2
 *          - ent_coef mean sum_k (ls_k + (1 + log 2 pi) / 2)
 * then the gradient of L (no gradient through an active log-std clamp),
 * scaled to 2-norm max_grad_norm when larger (max_grad_norm <= 0: never),
 * and one Adam step with bias correction:
 *   m = b1 m + (1 - b1) g;  v = b2 v + (1 - b2) g^2
 *   w -= lr (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) + adam_eps).
 * The two networks form one parameter vector for the norm and for Adam.
 *
 * Minibatches: epoch e permutes the M = T * N trajectory rows (row
 * r = t * N + i) by a four-round Feistel network on 2^b >= M codes (b even)
 * with cycle walking; round j maps (L, R) -> (R, L ^ F_j(R)) with F_j(R) the
 * first word of Philox4x32-10 at counter (R, j, e low, e high) and key (seed
 * low, seed high), masked to b/2 bits.  Minibatch j of epoch e takes the rows
 * at permutation positions j*B .. j*B + B - 1.
 *
 * Weight, gradient and moment vectors crossing this interface use the
 * env_set_weights layout of each network, [W1 | b1 | W2 | b2 | W3 | b3]
 * with W row-major [out][in]; a "parameter vector" is the policy's followed
 * by the value network's (ppo_param_counts gives the two lengths).
 * --------------------------------------------------------------------------- */
#define AUV_PPO_FP32 0u   /* GEMMs on the CUDA cores in fp32                     */
#define AUV_PPO_TF32 1u   /* GEMMs on the tensor cores, tf32 operands, fp32 sums */
#define AUV_PPO_BF16 2u   /* GEMMs on the tensor cores, bf16 operands, fp32 sums */
#define AUV_PPO_VALUE_ONLY 1u /* flags: train the value network alone on
 * L = vf_coef mean (V - ret)^2 / 2 (the critic regression of SHAC, whose
 * TD(lambda) targets are env_gae's returns); the policy is neither run nor
 * changed, and batch.act, .logp, .adv may be NULL. */
#define AUV_PPO_GEMM_PATH 2u /* flags: in bf16 mode, run the forward pass and
 * the input gradients as separate GEMMs (auv_gemm) and tanh passes.  Without
 * it a bf16 learner with hidden == 256, obs_dim <= 18 runs both networks'
 * forward passes and their backward-data (dL/dZ2, dL/dZ1 with the tanh
 * derivatives) on the tcgen05 engine of env_rollout (weights, and their
 * transposes, packed from the fp32 master copy every step; tanh on the fp32
 * pre-activation, each product rounded to bf16 once).  The weight gradients
 * are tcgen05 GEMMs over the minibatch (auv_gemm) in every mode.  All
 * products of every precision run in the library's own kernels. */
#define AUV_PPO_STATS 8   /* floats in a statistics record:                       */
/* [0] surrogate (policy) loss, [1] value loss (mean (V - ret)^2 / 2),
 * [2] entropy, [3] approx. KL mean(logp_old - logp), [4] clip fraction
 * mean(|r - 1| > clip_eps), [5] gradient norm before clipping, [6] total loss
 * L, [7] gradient steps the record covers.  ppo_update averages [0..6] over
 * its steps. */

typedef struct auv_ppo_config {
  uint32_t struct_size;   /* sizeof(auv_ppo_config)                          */
  uint32_t obs_dim;       /* network input width, 1 .. 64 (18 Fossen, 12 paper) */
  uint32_t act_dim;       /* A, 1 .. 8: the policy head is 2A wide            */
  uint32_t hidden;        /* H, a multiple of 8 in [8, 1024]                   */
  uint32_t minibatch;     /* B samples per gradient step, 2 .. 2^22            */
  uint32_t precision;     /* AUV_PPO_FP32 | AUV_PPO_TF32 | AUV_PPO_BF16        */
  uint32_t norm_adv;      /* 1: normalise advantages per minibatch, 0: not     */
  uint32_t flags;         /* AUV_PPO_VALUE_ONLY | AUV_PPO_GEMM_PATH, or 0      */
  uint64_t seed;          /* key of the minibatch permutations                 */
  float clip_eps;         /* > 0                                               */
  float vf_coef, ent_coef;            /* finite                                */
  float max_grad_norm;                /* <= 0: no clipping                     */
  float lr, adam_beta1, adam_beta2, adam_eps;   /* lr >= 0, betas in [0, 1), eps > 0 */
  float logstd_min, logstd_max;       /* the rollout's log-std clamp           */
} auv_ppo_config;

/* The trajectory a PPO update reads: the rollout's arrays (env_rollout with
 * obs, act and logp) and env_gae's advantages and returns.  Device memory,
 * 4-byte aligned, fp32.  obs [T][obs_dim][N], act [T][act_dim][N], logp, adv,
 * ret [T][N].  T, N >= 1 and T * N <= 2^31. */
typedef struct auv_ppo_batch {
  const float* obs;
  const float* act;
  const float* logp;
  const float* adv;
  const float* ret;
  uint32_t T, N;
} auv_ppo_batch;

typedef struct auv_ppo auv_ppo;

/* Create a learner on the current device: weights zero (call ppo_set_weights),
 * Adam moments zero, t = 0, epoch = 0.  AUV_ERR_INVALID on a bad config. */
int ppo_create(const auv_ppo_config* cfg, auv_ppo** out);
int ppo_destroy(auv_ppo* p);
const char* ppo_last_error(const auv_ppo* p);
int ppo_param_counts(const auv_ppo* p, uint64_t* n_policy, uint64_t* n_value);

/* Load both networks (device or host memory, env_set_weights layout) and
 * reset the Adam moments, t and epoch to 0.  Synchronises `stream`. */
int ppo_set_weights(auv_ppo* p, const float* policy, const float* value, void* stream);
/* Copy both networks out (device or host memory); synchronises `stream`. */
int ppo_get_weights(auv_ppo* p, float* policy, float* value, void* stream);

/* Adam state for checkpoints: moments m, v as parameter vectors (device or
 * host memory), the step count t and the next epoch number.  get
 * synchronises `stream`; set does too. */
int ppo_get_state(auv_ppo* p, float* m, float* v, uint64_t* t, uint64_t* epoch, void* stream);
int ppo_set_state(auv_ppo* p, const float* m, const float* v, uint64_t t, uint64_t epoch,
                  void* stream);

/*
 * ppo_grads: the gradient of L on minibatch `minibatch` of epoch `epoch`
 * (needs (minibatch + 1) * B <= T * N).  The gradient stays in the learner for
 * ppo_apply; if grad is not NULL it is also written there as a parameter
 * vector (device memory, 4-byte aligned), e.g. to be averaged over ranks
 * before ppo_apply.  If stats is not NULL (device memory, AUV_PPO_STATS
 * floats) the minibatch's record is written there ([5] = 0, [7] = 1).
 * Asynchronous on `stream`.
 */
int ppo_grads(auv_ppo* p, const auv_ppo_batch* batch, uint64_t epoch, uint32_t minibatch,
              float* grad, float* stats, void* stream);

/* ppo_apply: clip and take one Adam step (t += 1) with the learner's last
 * gradient (grad NULL) or with the parameter vector grad (device memory).
 * stats, if not NULL, receives the gradient norm in [5] (others untouched). */
int ppo_apply(auv_ppo* p, const float* grad, float* stats, void* stream);

/*
 * ppo_update: `epochs` passes over the batch, each of n_minibatches gradient
 * steps (minibatch j of epoch p->epoch, then p->epoch += 1), i.e. the whole
 * PPO update of one rollout; needs n_minibatches * B <= T * N.  stats, if not
 * NULL, receives the record averaged over the steps.  Asynchronous on
 * `stream`; the weights (ppo_get_weights, or the pointers of ppo_weights) are
 * the updated ones once it completes.  Each call first copies the batch into
 * a sample-major buffer (T * N rows of round8(obs_dim + act_dim + 3) floats,
 * one coalesced pass) from which every step gathers its minibatch; the
 * learner allocates that buffer the first time it sees a batch of more rows
 * than the last (the one allocation after ppo_create) and frees it in
 * ppo_destroy.  If the allocation fails the steps gather from the batch's
 * own arrays.
 */
int ppo_update(auv_ppo* p, const auv_ppo_batch* batch, uint32_t epochs, uint32_t n_minibatches,
               float* stats, void* stream);

/* ppo_status: synchronise `stream`, copy the learner's device status block
 * to *out and return out->code (the auv_status fields as for env_status):
 * AUV_ERR_TIMEOUT if a tensor-core engine launch of a gradient step gave up
 * on a bounded wait (the update's results are then invalid), AUV_OK
 * otherwise.  ppo_clear_status zeroes it (asynchronously on stream). */
int ppo_status(auv_ppo* p, auv_status* out, void* stream);
int ppo_clear_status(auv_ppo* p, void* stream);

/* ppo_export_weights: write both networks, in the env_set_weights layout,
 * to device memory (asynchronous on `stream`) -- e.g. straight into the
 * buffers an env_set_weights call then reads. */
int ppo_export_weights(auv_ppo* p, float* policy, float* value, void* stream);

/*
 * env_adjoint: reverse-mode adjoint of the control step over a window of
 * actions -- the back-propagation through the dynamics of SHAC (paper
 * §III-A, short-horizon actor-critic; Xu et al. 2022).  From each env's
 * current state x_0 = (p, q, nu) the window takes T control steps with the
 * given actions (the rollout's own step: allocation with clip, substeps,
 * reward, auto-reset) and forms
 *   J = sum_t coef[t] r_t + <lam_T, x_T>
 * with x_T the state after the last step.  Outputs dJ/da_t (grad_act) and
 * dJ/dx_0 (lam_0).  An episode end inside the window replaces the state by
 * its reset draw: nothing before it reaches later rewards or x_T.  The
 * clip's derivative is taken as 1 on [-1, 1] and 0 outside.
 * Shapes by model (A = env_layout's act_dim, S = the adjoint's state rows):
 *   Fossen: A = 8, S = 13 (p, q, nu; nu_prev is overwritten by every step);
 *   paper:  A = 6, S = 61 (p, q, nu and the 8 x 6 action-history rows of its
 *           state layout: the moving-average reward term makes an action
 *           reach later rewards through them).
 *   act [T][A][N], grad_act [T][A][N]: device memory.
 *   coef [T]: device memory.
 *   lam_T [S][N]: device memory, or NULL for 0.
 *   lam_0 [S][N], rew_out [T][N] (fp32), done_out [T][N] (u8): optional
 *   outputs, device or mapped page-locked host memory.
 * The env's state, episode counters and step counter are not changed (step
 * with env_step_actions to advance).  1 <= T <= AUV_ADJOINT_MAX_T; at most
 * AUV_ADJOINT_MAX_SUBSTEPS substeps (AUV_ERR_UNSUPPORTED).  The first call at
 * a given N * T allocates the window's scratch (30 floats per env-step plus
 * 61 per env) on the device.
 */
#define AUV_ADJOINT_MAX_T 64
#define AUV_ADJOINT_MAX_SUBSTEPS 8
int env_adjoint(auv_env* env, int T, const float* act, const float* coef, const float* lam_T,
                float* grad_act, float* lam_0, float* rew_out, uint8_t* done_out, void* stream);

/*
 * env_shac_window: SHAC's actor gradient over one window in closed loop
 * (paper §III-A: short-horizon actor-critic; Xu et al. 2022).  From each
 * env's current state the policy `policy` (env_set_weights layout,
 * obs -> hidden -> hidden -> 2A: means and log-stds of the A commands; the
 * Fossen model 18 -> .. -> 16, the paper model 12 -> .. -> 12) acts for
 * T steps with the reparameterised action a = mu + exp(clamp(ls)) eps (eps:
 * the rollout's action noise at the env's global steps), and the env
 * advances (state, counters, global step += T).  With the critic `value`
 * (same layout, head 1; NULL for none) at the observation after the last
 * step,
 *   J = sum over envs [ sum_t coef[t] r_t + coef_V V(o_T) ],
 * and grad (device memory, the policy's length) receives dJ/d(policy) by
 * back-propagation through the dynamics, the policy network and the
 * observation.  Gradients stop at the window's start and at episode ends
 * inside it (the state after an end is a reset draw).  Optional outputs:
 * J_out [N] each env's J; obs_out [T][obs][N] the observation of each step
 * (the rollout's layout: with rew_out, done_out [T][N], env_value and
 * env_gae it gives the critic's TD(lambda) targets); device or mapped
 * page-locked host memory for J_out, rew_out, done_out, device memory for
 * obs_out.  policy, value, coef [T], grad: device memory.
 * precision: AUV_PPO_FP32 (network products on the CUDA cores in fp32) or
 * AUV_PPO_TF32 (on the tensor cores, tf32 operands, fp32 sums); the physics
 * and its adjoint are fp32 either way.
 * Either model (the paper model's adjoint carries its action-history rows
 * between steps, as env_adjoint's does); 1 <= T <= AUV_ADJOINT_MAX_T, at most
 * AUV_ADJOINT_MAX_SUBSTEPS substeps, hidden a multiple of 8 up to 1024.
 * The first call at a given (N, T) allocates the window's workspace
 * (activations of every step: about T N (2 hidden + 80) floats).
 */
int env_shac_window(auv_env* env, const float* policy, const float* value, int T,
                    const float* coef, float coef_V, uint32_t precision, float* grad,
                    float* J_out, float* obs_out, float* rew_out, uint8_t* done_out,
                    void* stream);

/*
 * env_inverse_allocate: thruster commands for body-frame wrenches, the map
 * the paper's controllers go through at deployment (§V-B: the policy's
 * forces and torques -> individual thrusters through the allocation matrix).
 * With Bm = alloc * thrust_max (the env's 6 x 8 matrix), the commands are
 * the minimum-norm solution of Bm u = tau clipped to the thrusters' range:
 *   cmd = clip(pinv(Bm) tau, -1, 1)
 * (pinv = Bm^T (Bm Bm^T)^-1, formed once in double on the host).
 * wrench [6][n]: device memory; cmd [8][n]: device or mapped page-locked
 * host memory.  AUV_ERR_UNSUPPORTED if the allocation has rank < 6.
 * (The PWM interpolation after it is vehicle-specific and not built.)
 */
int env_inverse_allocate(auv_env* env, int n, const float* wrench, float* cmd, void* stream);

/* ---------------------------------------------------------------------------
 * Replay buffer for off-policy learning (DroQ, paper §III-A; Hiraoka et al.
 * 2022): a device ring of `capacity` transitions (obs, act, rew, next_obs,
 * done), stored sample-major.
 *
 * rbuf_insert adds a rollout's T x N transitions: transition (t, i) goes to
 * slot (head + t*N + i) mod capacity with obs = obs[t][.][i], act =
 * act[t][.][i], rew / done = [t][i], next_obs = obs[t+1][.][i] (last_obs for
 * t = T-1: the observation after the last step).  After an auto-reset the
 * next observation is the new episode's first: a time-limit end is stored
 * as a terminal transition (done = 1).  Inputs are the rollout's arrays in
 * device memory: obs [T][D][N], act [T][A][N], rew [T][N] fp32, done [T][N]
 * u8, last_obs [D][N].  head and size advance on the host at the call.
 *
 * rbuf_sample draws B transitions uniformly from the filled slots: sample b
 * of draw `draw` takes the first word w of Philox4x32-10 at counter
 * (b, 0x52420000, draw low, draw high) with key (seed low, seed high) and
 * reads slot floor(w * size / 2^32).  Outputs (device memory): obs and
 * next_obs [B][D], act [B][A], rew [B] fp32, done [B] u8, and optionally
 * the slots idx [B] (u32).  AUV_ERR_INVALID when the buffer is empty.
 * Both calls are asynchronous on `stream`; a sample sees every insert
 * issued before it on the same stream.
 * --------------------------------------------------------------------------- */
typedef struct auv_rbuf auv_rbuf;
int rbuf_create(uint32_t obs_dim, uint32_t act_dim, uint64_t capacity, auv_rbuf** out);
int rbuf_destroy(auv_rbuf* r);
const char* rbuf_last_error(const auv_rbuf* r);
int rbuf_size(const auv_rbuf* r, uint64_t* size, uint64_t* head);
int rbuf_insert(auv_rbuf* r, int T, int N, const float* obs, const float* act, const float* rew,
                const uint8_t* done, const float* last_obs, void* stream);
int rbuf_sample(auv_rbuf* r, uint32_t B, uint64_t seed, uint64_t draw, float* obs, float* act,
                float* rew, float* next_obs, uint8_t* done, uint32_t* idx, void* stream);

/* Global step counter (action-noise stream index) get/set, for checkpoints. */
int env_get_step(const auv_env* env, uint64_t* t_g);
int env_set_step(auv_env* env, uint64_t t_g);

/*
 * Snapshot of a batch for checkpoint and resume: everything that determines
 * the envs' future steps besides the configuration and the network weights.
 * Per env that is the dynamic state of the vehicle (the body pose and
 * velocities of §IV-B; the paper model adds the action history read by the
 * moving-average term of Eq. 7), the episode's randomised parameters (goal
 * of §V-A1, domain randomisation of §IV-C), the control steps taken in the
 * episode and the index of the next episode's reset draw; for the batch the
 * global step t_g that keys the action noise.  The arrays are caller-owned,
 * in the layout of auv_buffers (row counts from env_layout), device or host
 * memory (page-locked host memory keeps the copies asynchronous).
 */
typedef struct auv_snapshot {
  uint32_t struct_size;   /* sizeof(auv_snapshot): version guard            */
  uint32_t model;         /* AUV_MODEL_* of the env the snapshot came from  */
  uint32_t n_envs;        /* N                                              */
  uint32_t state_fields;  /* rows of state                                  */
  uint32_t param_fields;  /* rows of params                                 */
  uint32_t reserved;      /* 0                                              */
  uint64_t t_g;           /* global step (action-noise stream index)        */
  float* state;           /* [state_fields][N]                              */
  float* params;          /* [param_fields][N]                              */
  int32_t* t_ep;          /* [N]                                            */
  uint32_t* episode;      /* [N]                                            */
} auv_snapshot;

/*
 * env_get_state: copy the env's state, params, t_ep and episode arrays into
 * the snapshot's arrays (4-byte aligned, non-NULL) and fill its model,
 * n_envs, field counts and t_g.  The copies are enqueued on `stream` after
 * the work already there; t_g is the counter as of the call (it counts the
 * steps of every rollout enqueued before it).  The snapshot is complete when
 * `stream` has reached this point.
 * env_set_state: the reverse, into an env of the same model and n_envs:
 * copies the snapshot's arrays into the env's buffers on `stream` and sets
 * t_g.  Continuing from it reproduces, bit for bit, the steps the source env
 * would have taken next (same configuration and weights).
 * Errors: AUV_ERR_INVALID (NULL, struct_size, model, n_envs or field counts
 * that do not match the env), AUV_ERR_SIZE (misaligned array), AUV_ERR_CUDA.
 */
int env_get_state(auv_env* env, auv_snapshot* snap, void* stream);
int env_set_state(auv_env* env, const auv_snapshot* snap, void* stream);

/*
 * env_status: synchronise `stream`, copy the device status block to *out and
 * return out->code.  env_clear_status zeroes it (asynchronously on stream).
 */
int env_status(auv_env* env, auv_status* out, void* stream);
int env_clear_status(auv_env* env, void* stream);

/*
 * env_selftest_wait_timeout: failure-detection self-test.  Launches one
 * thread that waits, with the same bounded wait the tensor-core kernels use
 * on their mbarriers, on a barrier phase that nothing completes.  The wait
 * gives up after limit_us microseconds (1 .. 5e6) and latches AUV_ERR_TIMEOUT
 * and timeouts += 1 in the status block, read back by env_status; the CUDA
 * context stays usable.  (A library check, not part of the paper's method.)
 */
int env_selftest_wait_timeout(auv_env* env, uint32_t limit_us, void* stream);

/* ---------------------------------------------------------------------------
 * The learners' dense product (the contractions of the PPO update and of the
 * SHAC window, paper §III-A), on its own:
 *
 *   C[M][N] = beta * C + sum_{k < K} A(m, k) B(n, k)
 *
 * A(m, k) is A[m * lda + k] (a_mn = 0: rows are the M index, K contiguous)
 * or A[k * lda + m] (a_mn = 1: a sample-major array read along its samples,
 * as in a weight gradient); B(n, k) likewise with ldb, b_mn.  C is row-major
 * with ldc >= N, fp32, or bf16 with c_bf16 = 1 (bf16 precision only; rounded
 * to nearest even).  precision: AUV_PPO_BF16 (bf16 A and B, tcgen05
 * kind::f16), AUV_PPO_TF32 (fp32 A and B read as tf32, tcgen05 kind::tf32)
 * or AUV_PPO_FP32 (fp32 on CUDA cores); accumulation is fp32.  Tensor-core
 * precisions need A, B 16-byte aligned and lda, ldb times the element size a
 * multiple of 16 bytes (else AUV_ERR_SIZE).  workspace (device, or NULL):
 * room for the fp32 partials of a contraction split over CTAs, at least
 * auv_gemm_workspace_bytes(M, N, K) bytes for the split to be used;
 * partials are added in a fixed order, so results are reproducible.
 * status: a device auv_status the kernels latch AUV_ERR_TIMEOUT into if a
 * bounded wait gives up.  Asynchronous on stream.  Returns AUV_OK,
 * AUV_ERR_INVALID, AUV_ERR_SIZE or AUV_ERR_CUDA.
 * --------------------------------------------------------------------------- */
size_t auv_gemm_workspace_bytes(int M, int N, int K);
int auv_gemm(uint32_t precision, int M, int N, int K, const void* A, int lda, int a_mn,
             const void* B, int ldb, int b_mn, void* C, int ldc, int c_bf16, float beta,
             void* workspace, size_t workspace_bytes, auv_status* status, void* stream);

/* ---------------------------------------------------------------------------
 * Roofline probes (measurement helpers, not on any hot path).  Each enqueues
 * work of a known operation count on `stream`; the caller times it.
 *
 * auv_probe_ffma: blocks x threads threads, each running `iters` rounds of 8
 *   independent dependent FMAs: 16 * iters flop per thread (the FP32 pipe).
 * auv_probe_tanh: the same shape with tanh.approx.f32: 8 * iters operations
 *   per thread (the multi-function unit).
 * auv_probe_ex2: the same shape with ex2.approx.ftz.f32: 8 * iters operations
 *   per thread.
 *   blocks in [1, 65535], threads a multiple of 32 in [32, 1024], iters >= 1;
 *   sink: device memory (of the current device) of blocks * threads floats
 *   (written only to keep the work from being removed); a host pointer is
 *   AUV_ERR_INVALID.
 * auv_probe_gemm: one n x n x n cuBLAS GEMM, C = A B (column-major, fp32 C),
 *   with A, B fp32 and tf32 tensor-core math (AUV_PPO_TF32) or bf16 operands
 *   (AUV_PPO_BF16): 2 n^3 flop.  n a multiple of 16.
 * auv_probe_mma: `blocks` CTAs (one per SM), each issuing `iters` tcgen05
 *   MMAs of shape M = 128, N = n and K = 16 bf16 (kind::f16), or K = 8 tf32
 *   (kind::tf32) when tf32 is nonzero, fp32 accumulator; A in shared memory,
 *   or in tensor memory when a_tmem is nonzero; back to back from one
 *   thread, then one commit and one bounded wait.  cycles: device memory
 *   (of the current device) of `blocks` uint64 values, each the SM cycles
 *   from the first issue to the completion (0 if the wait gave up); a host
 *   pointer is AUV_ERR_INVALID.
 *   n in {16, 32, 64, 128, 256}, iters in [1, 2^20], blocks in [1, 65535].
 * Return AUV_OK, AUV_ERR_INVALID on bad arguments or AUV_ERR_CUDA.
 * --------------------------------------------------------------------------- */
int auv_probe_ffma(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream);
int auv_probe_tanh(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream);
int auv_probe_ex2(uint32_t blocks, uint32_t threads, uint32_t iters, float* sink, void* stream);
int auv_probe_mma(int n, int a_tmem, int tf32, uint32_t iters, uint32_t blocks, uint64_t* cycles,
                  void* stream);
int auv_probe_gemm(uint32_t precision, int n, const void* a, const void* b, void* c, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AUVENV_H */
