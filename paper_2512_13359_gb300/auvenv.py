"""Python binding of libauvenv.so (include/auvenv.h): argument marshalling only.

Every step of the rollout runs in the library's CUDA kernels; torch provides
device memory and streams.  There is no CPU fallback: if the library is
missing or cannot be loaded, LibraryMissing is raised.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from . import workloads as W

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libauvenv.so")

AUV_OK = 0
AUV_ERR_INVALID = -1
AUV_ERR_SIZE = -2
AUV_ERR_CUDA = -3
AUV_ERR_TIMEOUT = -4
AUV_ERR_NAN = -5
AUV_ERR_UNSUPPORTED = -6
AUV_MLP_FP32 = 0
AUV_MLP_BF16 = 1
AUV_MLP_TF32 = 2
AUV_MODEL_FOSSEN = 0
AUV_MODEL_PAPER = 1
AUV_PPO_FP32 = 0
AUV_PPO_TF32 = 1
AUV_PPO_BF16 = 2
AUV_PPO_STATS = 8
AUV_PPO_VALUE_ONLY = 1
AUV_PPO_GEMM_PATH = 2
PPO_PRECISION = {"fp32": AUV_PPO_FP32, "tf32": AUV_PPO_TF32, "bf16": AUV_PPO_BF16}
PPO_STAT_NAMES = ("pg_loss", "v_loss", "entropy", "approx_kl", "clip_frac", "grad_norm", "loss",
                  "steps")

EXPORTED = ("env_abi_version", "env_create", "env_destroy", "env_last_error", "env_set_weights",
            "env_reset", "env_rollout", "env_value", "env_step", "env_step_actions", "env_observe",
            "env_policy_forward", "env_draw_words", "env_get_step", "env_set_step",
            "env_get_state", "env_set_state",
            "env_status", "env_clear_status", "env_selftest_wait_timeout",
            "env_policy_forward_noalloc", "env_layout", "env_gae", "env_adjoint",
            "env_inverse_allocate", "env_shac_window", "rbuf_create", "rbuf_destroy", "rbuf_last_error",
            "rbuf_size", "rbuf_insert", "rbuf_sample",
            "ppo_create", "ppo_destroy", "ppo_last_error", "ppo_param_counts", "ppo_set_weights",
            "ppo_get_weights", "ppo_get_state", "ppo_set_state", "ppo_grads", "ppo_apply",
            "ppo_update", "ppo_export_weights", "ppo_status", "ppo_clear_status",
            "auv_gemm", "auv_gemm_workspace_bytes",
            "auv_probe_ffma", "auv_probe_tanh", "auv_probe_ex2", "auv_probe_mma", "auv_probe_gemm")


class LibraryMissing(RuntimeError):
    pass


class AuvError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"auvenv error {code}: {msg}")
        self.code = code


class AuvConfig(C.Structure):
    _fields_ = [
        ("struct_size", C.c_uint32), ("n_envs", C.c_uint32), ("substeps", C.c_uint32),
        ("episode_len", C.c_uint32), ("seed", C.c_uint32), ("env_id_base", C.c_uint32),
        ("dr_enable", C.c_uint32),
        ("dt", C.c_float), ("mass", C.c_float), ("inertia", C.c_float * 3),
        ("added_mass", C.c_float * 6), ("damp_lin", C.c_float * 6), ("damp_quad", C.c_float * 6),
        ("gravity", C.c_float * 3), ("thrust_max", C.c_float), ("alloc", C.c_float * 48),
        ("w_pos", C.c_float), ("w_att", C.c_float), ("w_act", C.c_float), ("w_vs", C.c_float),
        ("init_pos_range", C.c_float), ("init_att_range", C.c_float),
        ("goal_pos_range", C.c_float), ("goal_yaw_range", C.c_float),
        ("current_range", C.c_float), ("dr_scale_lo", C.c_float), ("dr_scale_hi", C.c_float),
        ("dr_buoy_range", C.c_float), ("dr_cob_range", C.c_float),
        ("hidden", C.c_uint32), ("policy_out", C.c_uint32), ("mlp_mode", C.c_uint32),
        ("has_value", C.c_uint32), ("logstd_fixed", C.c_float * 8),
        ("logstd_min", C.c_float), ("logstd_max", C.c_float),
        ("model", C.c_uint32), ("f_max", C.c_float), ("tau_max", C.c_float),
        ("fluid_density", C.c_float), ("fluid_viscosity", C.c_float), ("g_eff", C.c_float),
        ("dr_gravity_range", C.c_float), ("goal_att_range", C.c_float),
        ("w_axes", C.c_float * 3), ("w_vel", C.c_float), ("w_mavg", C.c_float),
        ("mavg_len", C.c_uint32),
    ]


class AuvLayout(C.Structure):
    _fields_ = [("obs_dim", C.c_uint32), ("act_dim", C.c_uint32), ("state_fields", C.c_uint32),
                ("param_fields", C.c_uint32)]


class AuvBuffers(C.Structure):
    _fields_ = [("state", C.c_void_p), ("params", C.c_void_p), ("t_ep", C.c_void_p),
                ("episode", C.c_void_p)]


class AuvTraj(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("act", C.c_void_p), ("logp", C.c_void_p),
                ("value", C.c_void_p), ("rew", C.c_void_p), ("done", C.c_void_p)]


class PpoConfig(C.Structure):
    _fields_ = [
        ("struct_size", C.c_uint32), ("obs_dim", C.c_uint32), ("act_dim", C.c_uint32),
        ("hidden", C.c_uint32), ("minibatch", C.c_uint32), ("precision", C.c_uint32),
        ("norm_adv", C.c_uint32), ("flags", C.c_uint32), ("seed", C.c_uint64),
        ("clip_eps", C.c_float), ("vf_coef", C.c_float), ("ent_coef", C.c_float),
        ("max_grad_norm", C.c_float), ("lr", C.c_float), ("adam_beta1", C.c_float),
        ("adam_beta2", C.c_float), ("adam_eps", C.c_float), ("logstd_min", C.c_float),
        ("logstd_max", C.c_float)]


class PpoBatch(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("act", C.c_void_p), ("logp", C.c_void_p),
                ("adv", C.c_void_p), ("ret", C.c_void_p), ("T", C.c_uint32), ("N", C.c_uint32)]


class AuvSnapshot(C.Structure):
    _fields_ = [("struct_size", C.c_uint32), ("model", C.c_uint32), ("n_envs", C.c_uint32),
                ("state_fields", C.c_uint32), ("param_fields", C.c_uint32),
                ("reserved", C.c_uint32), ("t_g", C.c_uint64), ("state", C.c_void_p),
                ("params", C.c_void_p), ("t_ep", C.c_void_p), ("episode", C.c_void_p)]


class AuvStatus(C.Structure):
    _fields_ = [("code", C.c_int32), ("nan_flag", C.c_int32), ("first_nan_env", C.c_int32),
                ("timeouts", C.c_int32)]


_lib = None


def lib(path: str | None = None):
    """Load libauvenv.so (once).  Raises LibraryMissing if absent."""
    global _lib
    if _lib is not None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise LibraryMissing(f"{p} not built; run paper_2512_13359_gb300.build.build()")
    try:
        L = C.CDLL(p)
    except OSError as e:
        raise LibraryMissing(f"cannot load {p}: {e}") from e
    P, I = C.c_void_p, C.c_int
    L.env_abi_version.restype = I
    L.env_create.argtypes = [P, P, C.POINTER(P)]
    L.env_destroy.argtypes = [P]
    L.env_last_error.argtypes = [P]
    L.env_last_error.restype = C.c_char_p
    L.env_set_weights.argtypes = [P, P, P, P]
    L.env_reset.argtypes = [P, P, P]
    L.env_rollout.argtypes = [P, I, P, P]
    L.env_value.argtypes = [P, P, I, P, P]
    L.env_step.argtypes = [P, P, P, P, P]
    L.env_step_actions.argtypes = [P, P, I, P, P, P, P]
    L.env_observe.argtypes = [P, P, P]
    L.env_policy_forward.argtypes = [P, P, I, P, P, P]
    L.env_draw_words.argtypes = [P, C.c_uint32, C.c_uint64, I, P, P]
    L.env_get_step.argtypes = [P, C.POINTER(C.c_uint64)]
    L.env_set_step.argtypes = [P, C.c_uint64]
    L.env_get_state.argtypes = [P, C.POINTER(AuvSnapshot), P]
    L.env_set_state.argtypes = [P, C.POINTER(AuvSnapshot), P]
    L.env_status.argtypes = [P, C.POINTER(AuvStatus), P]
    L.env_clear_status.argtypes = [P, P]
    L.env_selftest_wait_timeout.argtypes = [P, C.c_uint32, P]
    L.env_policy_forward_noalloc.argtypes = [I, I, P, P, P, I, P, P, P, P]
    L.env_layout.argtypes = [C.c_uint32, C.POINTER(AuvLayout)]
    L.env_gae.argtypes = [P, I, P, P, P, P, C.c_float, C.c_float, P, P, P]
    L.env_adjoint.argtypes = [P, I, P, P, P, P, P, P, P, P]
    L.env_inverse_allocate.argtypes = [P, I, P, P, P]
    L.env_shac_window.argtypes = [P, P, P, I, P, C.c_float, C.c_uint32, P, P, P, P, P, P]
    L.rbuf_create.argtypes = [C.c_uint32, C.c_uint32, C.c_uint64, C.POINTER(P)]
    L.rbuf_destroy.argtypes = [P]
    L.rbuf_last_error.argtypes = [P]
    L.rbuf_last_error.restype = C.c_char_p
    L.rbuf_size.argtypes = [P, C.POINTER(C.c_uint64), C.POINTER(C.c_uint64)]
    L.rbuf_insert.argtypes = [P, I, I, P, P, P, P, P, P]
    L.rbuf_sample.argtypes = [P, C.c_uint32, C.c_uint64, C.c_uint64, P, P, P, P, P, P, P]
    U64, U32 = C.c_uint64, C.c_uint32
    L.ppo_create.argtypes = [C.POINTER(PpoConfig), C.POINTER(P)]
    L.ppo_destroy.argtypes = [P]
    L.ppo_last_error.argtypes = [P]
    L.ppo_last_error.restype = C.c_char_p
    L.ppo_param_counts.argtypes = [P, C.POINTER(U64), C.POINTER(U64)]
    L.ppo_set_weights.argtypes = [P, P, P, P]
    L.ppo_get_weights.argtypes = [P, P, P, P]
    L.ppo_export_weights.argtypes = [P, P, P, P]
    L.ppo_get_state.argtypes = [P, P, P, C.POINTER(U64), C.POINTER(U64), P]
    L.ppo_set_state.argtypes = [P, P, P, U64, U64, P]
    L.ppo_grads.argtypes = [P, C.POINTER(PpoBatch), U64, U32, P, P, P]
    L.ppo_apply.argtypes = [P, P, P, P]
    L.ppo_update.argtypes = [P, C.POINTER(PpoBatch), U32, U32, P, P]
    L.ppo_status.argtypes = [P, C.POINTER(AuvStatus), P]
    L.auv_probe_ffma.argtypes = [U32, U32, U32, P, P]
    L.auv_probe_tanh.argtypes = [U32, U32, U32, P, P]
    L.auv_probe_ex2.argtypes = [U32, U32, U32, P, P]
    L.auv_probe_mma.argtypes = [I, I, I, U32, U32, P, P]
    L.auv_probe_gemm.argtypes = [U32, I, P, P, P, P]
    L.auv_gemm_workspace_bytes.argtypes = [I, I, I]
    L.auv_gemm_workspace_bytes.restype = C.c_size_t
    L.auv_gemm.argtypes = [U32, I, I, I, P, I, I, P, I, I, P, I, I, C.c_float, P, C.c_size_t, P,
                           P]
    L.ppo_clear_status.argtypes = [P, P]
    for name in EXPORTED:
        getattr(L, name).restype = getattr(L, name).restype or I
    L.env_last_error.restype = C.c_char_p
    L.ppo_last_error.restype = C.c_char_p
    L.rbuf_last_error.restype = C.c_char_p
    _lib = L
    return L


def make_config(w: dict) -> AuvConfig:
    c = AuvConfig()
    c.struct_size = C.sizeof(AuvConfig)
    c.n_envs = int(w["n_envs"])
    c.substeps = int(w["substeps"])
    c.episode_len = int(w["episode_len"])
    c.seed = int(w["seed"]) & 0xFFFFFFFF
    c.env_id_base = int(w.get("env_id_base", 0))
    c.dr_enable = int(w["dr_enable"])
    c.dt = float(w["dt"])
    c.mass = float(w["mass"])
    c.inertia[:] = [float(x) for x in w["inertia"]]
    c.added_mass[:] = [float(x) for x in w["added_mass"]]
    c.damp_lin[:] = [float(x) for x in w["damp_lin"]]
    c.damp_quad[:] = [float(x) for x in w["damp_quad"]]
    c.gravity[:] = [float(x) for x in w["gravity"]]
    c.thrust_max = float(w["thrust_max"])
    c.alloc[:] = [float(x) for x in np.asarray(w["alloc"], dtype=np.float64).reshape(-1)]
    for k in ("w_pos", "w_att", "w_act", "w_vs", "init_pos_range", "init_att_range",
              "goal_pos_range", "goal_yaw_range", "current_range", "dr_scale_lo", "dr_scale_hi",
              "dr_buoy_range", "dr_cob_range", "logstd_min", "logstd_max"):
        setattr(c, k, float(w[k]))
    c.hidden = int(w["hidden"])
    c.policy_out = int(w["policy_out"])
    c.mlp_mode = {"bf16": AUV_MLP_BF16, "tf32": AUV_MLP_TF32}.get(w["mlp"], AUV_MLP_FP32)
    c.has_value = int(w["has_value"])
    ls = [float(x) for x in w["logstd_fixed"]]
    c.logstd_fixed[:] = ls + [0.0] * (8 - len(ls))
    c.model = AUV_MODEL_PAPER if W.is_paper(w) else AUV_MODEL_FOSSEN
    for k in ("f_max", "tau_max", "fluid_density", "fluid_viscosity", "g_eff",
              "dr_gravity_range", "goal_att_range", "w_vel", "w_mavg"):
        setattr(c, k, float(w.get(k, 0.0)))
    c.w_axes[:] = [float(x) for x in w.get("w_axes", (1.0, 1.0, 1.0))]
    c.mavg_len = int(w.get("mavg_len", 1))
    return c


def layout(model: int) -> AuvLayout:
    out = AuvLayout()
    rc = lib().env_layout(int(model), C.byref(out))
    if rc != AUV_OK:
        raise AuvError(rc, lib().env_last_error(None).decode())
    return out


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream):
    import torch
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


class Env:
    """A batch of N environments on the current CUDA device.

    State lives in caller-owned torch tensors (SoA): state[S][N], params[P][N]
    (S, P = 19, 17 for the Fossen model, 61, 8 for the paper model), t_ep[N]
    (int32), episode[N] (int32 storage of uint32)."""

    def __init__(self, workload: dict, device=None):
        import torch
        self.w = dict(workload)
        self.n = int(workload["n_envs"])
        self.device = torch.device(device or "cuda")
        L = lib()
        n = self.n
        with torch.cuda.device(self.device):
            self.state = torch.zeros((W.state_fields(workload), n), dtype=torch.float32,
                                     device=self.device)
            self.params = torch.zeros((W.param_fields(workload), n), dtype=torch.float32,
                                      device=self.device)
            self.t_ep = torch.zeros(n, dtype=torch.int32, device=self.device)
            self.episode = torch.zeros(n, dtype=torch.int32, device=self.device)
            self.cfg = make_config(workload)
            bufs = AuvBuffers(self.state.data_ptr(), self.params.data_ptr(),
                              self.t_ep.data_ptr(), self.episode.data_ptr())
            h = C.c_void_p()
            rc = L.env_create(C.byref(self.cfg), C.byref(bufs), C.byref(h))
            if rc != AUV_OK:
                raise AuvError(rc, L.env_last_error(None).decode())
        self.h = h

    # -- helpers -------------------------------------------------------------
    def _check(self, rc):
        if rc != AUV_OK:
            raise AuvError(rc, lib().env_last_error(self.h).decode())

    def close(self):
        if getattr(self, "h", None):
            lib().env_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- entry points ----------------------------------------------------------
    def set_weights(self, policy, value=None, stream=None):
        """policy/value: torch tensors (host or device) or numpy float32 arrays."""
        keep = []

        def addr(x):
            if x is None:
                return None
            if isinstance(x, np.ndarray):
                a = np.ascontiguousarray(x, dtype=np.float32)
                keep.append(a)
                return a.ctypes.data_as(C.c_void_p)
            x = x.contiguous()
            keep.append(x)
            return C.c_void_p(x.data_ptr())

        self._check(lib().env_set_weights(self.h, addr(policy), addr(value), _stream(stream)))

    def reset(self, mask=None, stream=None):
        self._check(lib().env_reset(self.h, _ptr(mask), _stream(stream)))

    def rollout(self, T: int, traj: dict, stream=None):
        t = AuvTraj(*(traj.get(k).data_ptr() if traj.get(k) is not None else None
                      for k in ("obs", "act", "logp", "value", "rew", "done")))
        self._check(lib().env_rollout(self.h, int(T), C.byref(t), _stream(stream)))

    def value(self, obs, value, stream=None):
        """Value network on trajectory-layout observations obs[T][obs_dim][N] -> value[T][N]."""
        self._check(lib().env_value(self.h, _ptr(obs), int(obs.shape[0]), _ptr(value),
                                    _stream(stream)))

    def gae(self, rew, done, value, last_value, gamma, lam, adv, ret, stream=None):
        """Generalised advantage estimation over [T][N] trajectory arrays."""
        self._check(lib().env_gae(self.h, int(rew.shape[0]), _ptr(rew), _ptr(done), _ptr(value),
                                  _ptr(last_value), float(gamma), float(lam), _ptr(adv),
                                  _ptr(ret), _stream(stream)))

    def adjoint(self, act, coef, grad_act, lam_T=None, lam_0=None, rew=None, done=None,
                stream=None):
        """Reverse-mode adjoint of an action window from the current state
        (env_adjoint): fills grad_act [T][8][N] and, if given, lam_0 [13][N],
        rew and done [T][N]."""
        T = act.shape[0]
        self._check(lib().env_adjoint(self.h, T, _ptr(act), _ptr(coef), _ptr(lam_T),
                                      _ptr(grad_act), _ptr(lam_0), _ptr(rew), _ptr(done),
                                      _stream(stream)))

    def shac_window(self, policy, value, coef, coef_V, grad, J=None, rew=None, done=None,
                    obs=None, precision="fp32", stream=None):
        """SHAC actor gradient over a window of len(coef) steps in closed loop
        (env_shac_window); the env advances."""
        self._check(lib().env_shac_window(self.h, _ptr(policy), _ptr(value), coef.shape[0],
                                          _ptr(coef), float(coef_V), PPO_PRECISION[precision],
                                          _ptr(grad), _ptr(J), _ptr(obs), _ptr(rew), _ptr(done),
                                          _stream(stream)))

    def inverse_allocate(self, wrench, cmd, stream=None):
        """Thruster commands cmd [8][n] for wrenches [6][n] (env_inverse_allocate)."""
        self._check(lib().env_inverse_allocate(self.h, wrench.shape[1], _ptr(wrench), _ptr(cmd),
                                               _stream(stream)))

    def step(self, obs=None, rew=None, done=None, stream=None):
        self._check(lib().env_step(self.h, _ptr(obs), _ptr(rew), _ptr(done), _stream(stream)))

    def step_actions(self, act, rew, done, trace=None, stream=None):
        T = act.shape[0]
        self._check(lib().env_step_actions(self.h, _ptr(act), int(T), _ptr(rew), _ptr(done),
                                           _ptr(trace), _stream(stream)))

    def observe(self, out, stream=None):
        self._check(lib().env_observe(self.h, _ptr(out), _stream(stream)))

    def policy_forward(self, obs, head, value=None, stream=None):
        self._check(lib().env_policy_forward(self.h, _ptr(obs), int(obs.shape[0]), _ptr(head),
                                             _ptr(value), _stream(stream)))

    def draw_words(self, stream_id: int, index: int, n_blocks: int, out, stream=None):
        self._check(lib().env_draw_words(self.h, int(stream_id), int(index), int(n_blocks),
                                         _ptr(out), _stream(stream)))

    @property
    def t_g(self) -> int:
        v = C.c_uint64()
        self._check(lib().env_get_step(self.h, C.byref(v)))
        return int(v.value)

    @t_g.setter
    def t_g(self, value: int):
        self._check(lib().env_set_step(self.h, int(value)))

    def status(self, stream=None) -> AuvStatus:
        s = AuvStatus()
        lib().env_status(self.h, C.byref(s), _stream(stream))
        return s

    def get_state(self, snap: dict, stream=None) -> int:
        """env_get_state into snap's tensors (keys state, params, t_ep,
        episode; device or host).  Returns the snapshot's t_g."""
        sn = AuvSnapshot(C.sizeof(AuvSnapshot), 0, 0, 0, 0, 0, 0,
                         *(snap[k].data_ptr() for k in ("state", "params", "t_ep", "episode")))
        self._check(lib().env_get_state(self.h, C.byref(sn), _stream(stream)))
        snap.update(t_g=int(sn.t_g), model=int(sn.model), n_envs=int(sn.n_envs),
                    state_fields=int(sn.state_fields), param_fields=int(sn.param_fields))
        return int(sn.t_g)

    def set_state(self, snap: dict, stream=None):
        """env_set_state from snap's tensors, t_g and header fields (model,
        n_envs, field counts; as get_state filled them, else this env's)."""
        lay = AuvLayout()
        lib().env_layout(self.cfg.model, C.byref(lay))
        sn = AuvSnapshot(C.sizeof(AuvSnapshot), snap.get("model", self.cfg.model),
                         snap.get("n_envs", self.n), snap.get("state_fields", lay.state_fields),
                         snap.get("param_fields", lay.param_fields), 0, int(snap["t_g"]),
                         *(snap[k].data_ptr() for k in ("state", "params", "t_ep", "episode")))
        self._check(lib().env_set_state(self.h, C.byref(sn), _stream(stream)))

    def selftest_wait_timeout(self, limit_us: int, stream=None):
        self._check(lib().env_selftest_wait_timeout(self.h, int(limit_us), _stream(stream)))

    def clear_status(self, stream=None):
        self._check(lib().env_clear_status(self.h, _stream(stream)))

    # -- allocation helpers ----------------------------------------------------
    def alloc_traj(self, T: int, keys=("obs", "act", "logp", "value", "rew", "done"),
                   pinned_host: bool = False) -> dict:
        import torch
        n = self.n
        shapes = dict(obs=(T, W.obs_dim(self.w), n), act=(T, W.act_dim(self.w), n), logp=(T, n),
                      value=(T, n), rew=(T, n), done=(T, n))
        out = {}
        for k in keys:
            if k == "value" and not self.w["has_value"]:
                continue
            dt = torch.uint8 if k == "done" else torch.float32
            if pinned_host:
                out[k] = torch.empty(shapes[k], dtype=dt, pin_memory=True)
            else:
                out[k] = torch.empty(shapes[k], dtype=dt, device=self.device)
        return out


PPO_DEFAULTS = dict(clip_eps=0.2, vf_coef=0.5, ent_coef=0.0, max_grad_norm=0.5, lr=3e-4,
                    adam_beta1=0.9, adam_beta2=0.999, adam_eps=1e-8, logstd_min=-5.0,
                    logstd_max=2.0, norm_adv=True)


def make_ppo_config(obs_dim: int, act_dim: int, hidden: int, minibatch: int,
                    precision: str = "fp32", seed: int = 0, **hp) -> PpoConfig:
    h = dict(PPO_DEFAULTS, **hp)
    c = PpoConfig()
    c.struct_size = C.sizeof(PpoConfig)
    c.obs_dim, c.act_dim, c.hidden, c.minibatch = obs_dim, act_dim, hidden, minibatch
    c.precision = PPO_PRECISION[precision] if isinstance(precision, str) else int(precision)
    c.norm_adv = 1 if h.pop("norm_adv") else 0
    c.flags = ((AUV_PPO_VALUE_ONLY if h.pop("value_only", False) else 0)
               | (AUV_PPO_GEMM_PATH if h.pop("gemm_path", False) else 0))
    c.seed = seed
    for k, v in h.items():
        setattr(c, k, float(v))
    return c


class Learner:
    """PPO learner (include/auvenv.h, ppo_*) on the current CUDA device.

    Trajectory arguments are dicts of CUDA tensors in the rollout's layout:
    obs [T][obs_dim][N], act [T][act_dim][N], logp, adv, ret [T][N]."""

    def __init__(self, obs_dim: int, act_dim: int, hidden: int, minibatch: int,
                 precision: str = "fp32", seed: int = 0, **hp):
        import torch
        self.cfg = make_ppo_config(obs_dim, act_dim, hidden, minibatch, precision, seed, **hp)
        self.device = torch.device("cuda", torch.cuda.current_device())
        L = lib()
        h = C.c_void_p()
        rc = L.ppo_create(C.byref(self.cfg), C.byref(h))
        if rc != AUV_OK:
            raise AuvError(rc, L.ppo_last_error(None).decode())
        self.h = h
        a, b = C.c_uint64(), C.c_uint64()
        self._check(L.ppo_param_counts(h, C.byref(a), C.byref(b)))
        self.n_policy, self.n_value = a.value, b.value

    def _check(self, rc):
        if rc != AUV_OK:
            raise AuvError(rc, lib().ppo_last_error(self.h).decode())

    def close(self):
        if getattr(self, "h", None):
            lib().ppo_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @staticmethod
    def _batch(traj):
        """obs, ret required; act, logp, adv may be absent (value-only learner)."""
        T, N = traj["ret"].shape
        for k in ("obs", "act", "logp", "adv", "ret"):
            if traj.get(k) is not None and not traj[k].is_contiguous():
                raise ValueError(f"{k} must be contiguous")
        ptr = lambda k: traj[k].data_ptr() if traj.get(k) is not None else None
        return PpoBatch(ptr("obs"), ptr("act"), ptr("logp"), ptr("adv"), ptr("ret"), T, N)

    def set_weights(self, policy, value, stream=None):
        p = np.ascontiguousarray(policy, dtype=np.float32)
        v = np.ascontiguousarray(value, dtype=np.float32)
        if p.size != self.n_policy or v.size != self.n_value:
            raise ValueError("weight vector lengths do not match the networks")
        self._check(lib().ppo_set_weights(self.h, p.ctypes.data_as(C.c_void_p),
                                          v.ctypes.data_as(C.c_void_p), _stream(stream)))

    def get_weights(self, stream=None):
        p = np.empty(self.n_policy, dtype=np.float32)
        v = np.empty(self.n_value, dtype=np.float32)
        self._check(lib().ppo_get_weights(self.h, p.ctypes.data_as(C.c_void_p),
                                          v.ctypes.data_as(C.c_void_p), _stream(stream)))
        return p, v

    def export_weights(self, policy, value, stream=None):
        self._check(lib().ppo_export_weights(self.h, _ptr(policy), _ptr(value), _stream(stream)))

    def get_state(self, stream=None):
        n = self.n_policy + self.n_value
        m = np.empty(n, dtype=np.float32)
        v = np.empty(n, dtype=np.float32)
        t, e = C.c_uint64(), C.c_uint64()
        self._check(lib().ppo_get_state(self.h, m.ctypes.data_as(C.c_void_p),
                                        v.ctypes.data_as(C.c_void_p), C.byref(t), C.byref(e),
                                        _stream(stream)))
        return dict(m=m, v=v, t=t.value, epoch=e.value)

    def set_state(self, state, stream=None):
        m = np.ascontiguousarray(state["m"], dtype=np.float32)
        v = np.ascontiguousarray(state["v"], dtype=np.float32)
        self._check(lib().ppo_set_state(self.h, m.ctypes.data_as(C.c_void_p),
                                        v.ctypes.data_as(C.c_void_p), int(state["t"]),
                                        int(state["epoch"]), _stream(stream)))

    def grads(self, traj, epoch: int, minibatch: int, grad=None, stats=None, stream=None):
        b = self._batch(traj)
        self._check(lib().ppo_grads(self.h, C.byref(b), epoch, minibatch, _ptr(grad), _ptr(stats),
                                    _stream(stream)))

    def apply(self, grad=None, stats=None, stream=None):
        self._check(lib().ppo_apply(self.h, _ptr(grad), _ptr(stats), _stream(stream)))

    def update(self, traj, epochs: int, n_minibatches: int, stats=None, stream=None):
        b = self._batch(traj)
        self._check(lib().ppo_update(self.h, C.byref(b), epochs, n_minibatches, _ptr(stats),
                                     _stream(stream)))

    def status(self, stream=None) -> AuvStatus:
        """Synchronise and read the device status block (code 0: no engine
        wait gave up)."""
        s = AuvStatus()
        lib().ppo_status(self.h, C.byref(s), _stream(stream))
        return s

    def clear_status(self, stream=None):
        self._check(lib().ppo_clear_status(self.h, _stream(stream)))


def _probe_check(rc, what):
    if rc != AUV_OK:
        raise AuvError(rc, f"{what} failed")


def probe_ffma(blocks: int, threads: int, iters: int, sink, stream=None) -> int:
    """Enqueue the FFMA-chain probe; returns its flop count (16 per thread-iteration)."""
    _probe_check(lib().auv_probe_ffma(blocks, threads, iters, _ptr(sink), _stream(stream)), "ffma probe")
    return 16 * blocks * threads * iters


def probe_tanh(blocks: int, threads: int, iters: int, sink, stream=None) -> int:
    """Enqueue the tanh.approx.f32 probe; returns its operation count."""
    _probe_check(lib().auv_probe_tanh(blocks, threads, iters, _ptr(sink), _stream(stream)), "tanh probe")
    return 8 * blocks * threads * iters


def probe_ex2(blocks: int, threads: int, iters: int, sink, stream=None) -> int:
    """Enqueue the ex2.approx.ftz.f32 probe; returns its operation count."""
    _probe_check(lib().auv_probe_ex2(blocks, threads, iters, _ptr(sink), _stream(stream)), "ex2 probe")
    return 8 * blocks * threads * iters


def probe_mma(n: int, a_tmem: bool, iters: int, cycles, stream=None, tf32: bool = False) -> None:
    """Enqueue the tcgen05 MMA probe (bf16, or tf32 with tf32=True) on
    cycles.numel() CTAs (cycles: 64-bit device tensor, one SM-cycle span per
    CTA, 0 where the wait gave up)."""
    _probe_check(lib().auv_probe_mma(n, 1 if a_tmem else 0, 1 if tf32 else 0, iters,
                                     int(cycles.numel()), _ptr(cycles), _stream(stream)),
                 "mma probe")


def probe_gemm(precision: str, a, b, c, stream=None) -> int:
    """Enqueue one n x n x n cuBLAS GEMM (tf32 on fp32 operands, or bf16); returns 2 n^3."""
    n = int(a.shape[0])
    _probe_check(lib().auv_probe_gemm(PPO_PRECISION[precision], n, _ptr(a), _ptr(b), _ptr(c),
                                      _stream(stream)), "gemm probe")
    return 2 * n ** 3


class ReplayBuffer:
    """Device replay buffer (include/auvenv.h, rbuf_*) on the current device."""

    def __init__(self, obs_dim: int, act_dim: int, capacity: int):
        L = lib()
        h = C.c_void_p()
        rc = L.rbuf_create(obs_dim, act_dim, capacity, C.byref(h))
        if rc != AUV_OK:
            raise AuvError(rc, L.rbuf_last_error(None).decode())
        self.h = h
        self.obs_dim, self.act_dim, self.capacity = obs_dim, act_dim, capacity

    def _check(self, rc):
        if rc != AUV_OK:
            raise AuvError(rc, lib().rbuf_last_error(self.h).decode())

    def close(self):
        if getattr(self, "h", None):
            lib().rbuf_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    @property
    def size(self):
        a, b = C.c_uint64(), C.c_uint64()
        self._check(lib().rbuf_size(self.h, C.byref(a), C.byref(b)))
        return a.value, b.value

    def insert(self, obs, act, rew, done, last_obs, stream=None):
        T, _, N = obs.shape
        self._check(lib().rbuf_insert(self.h, T, N, _ptr(obs), _ptr(act), _ptr(rew), _ptr(done),
                                      _ptr(last_obs), _stream(stream)))

    def sample(self, B: int, seed: int, draw: int, out=None, with_idx=False, stream=None):
        import torch
        if out is None:
            out = dict(obs=torch.empty((B, self.obs_dim), device="cuda"),
                       act=torch.empty((B, self.act_dim), device="cuda"),
                       rew=torch.empty(B, device="cuda"),
                       next_obs=torch.empty((B, self.obs_dim), device="cuda"),
                       done=torch.empty(B, dtype=torch.uint8, device="cuda"))
            if with_idx:
                out["idx"] = torch.empty(B, dtype=torch.int32, device="cuda")
        self._check(lib().rbuf_sample(self.h, B, seed, draw, _ptr(out["obs"]), _ptr(out["act"]),
                                      _ptr(out["rew"]), _ptr(out["next_obs"]), _ptr(out["done"]),
                                      _ptr(out.get("idx")), _stream(stream)))
        return out


def gemm(precision: str, M: int, N: int, K: int, A, lda: int, a_mn: bool, B, ldb: int,
         b_mn: bool, Cout, ldc: int, beta: float = 0.0, workspace=None, status=None,
         stream=None):
    """auv_gemm on torch device tensors: Cout[M][N] = beta Cout + A B^T with
    A(m, k) = A[m*lda + k] (a_mn False) or A[k*lda + m] (a_mn True), B
    likewise.  precision 'bf16' | 'tf32' | 'fp32'; Cout fp32 or bf16.
    status: int32 device tensor of 4 (allocated if None).  Returns status."""
    import torch
    if status is None:
        status = torch.zeros(4, dtype=torch.int32, device=Cout.device)
    ws_ptr = C.c_void_p(workspace.data_ptr()) if workspace is not None else None
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = lib().auv_gemm(PPO_PRECISION[precision], M, N, K, C.c_void_p(A.data_ptr()), lda,
                        int(a_mn), C.c_void_p(B.data_ptr()), ldb, int(b_mn),
                        C.c_void_p(Cout.data_ptr()), ldc, int(Cout.dtype == torch.bfloat16),
                        float(beta), ws_ptr, ws_bytes, C.c_void_p(status.data_ptr()),
                        _stream(stream))
    if rc != AUV_OK:
        raise AuvError(rc, "auv_gemm")
    return status
