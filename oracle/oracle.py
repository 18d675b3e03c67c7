"""ctypes loader for the CPU oracle (oracle/auv_oracle.cpp).

TEST INFRASTRUCTURE: only tests/, __graft_entry__.smoke() and the CPU-baseline
leg of bench.py may import this module.  It never touches the CUDA library.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "auv_oracle.cpp")
LIB = os.path.join(HERE, "liboracle.so")


def build(force: bool = False) -> str:
    """Compile the oracle: plain C++17, -O2, no FMA contraction."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        cmd = ["g++", "-std=c++17", "-O2", "-ffp-contract=off", "-fno-fast-math",
               "-shared", "-fPIC", "-o", LIB + ".tmp", SRC]
        subprocess.check_call(cmd)
        os.replace(LIB + ".tmp", LIB)
    return LIB


class OracleModel(C.Structure):
    _fields_ = [
        ("n_substeps", C.c_int32), ("episode_len", C.c_int32), ("seed", C.c_uint32),
        ("dr_enable", C.c_int32),
        ("dt", C.c_double), ("mass", C.c_double), ("inertia", C.c_double * 3),
        ("added_mass", C.c_double * 6), ("damp_lin", C.c_double * 6),
        ("damp_quad", C.c_double * 6), ("gravity", C.c_double * 3),
        ("thrust_max", C.c_double), ("alloc", C.c_double * 48),
        ("w_pos", C.c_double), ("w_att", C.c_double), ("w_act", C.c_double),
        ("w_vs", C.c_double),
        ("init_pos_range", C.c_float), ("init_att_range", C.c_float),
        ("goal_pos_range", C.c_float), ("goal_yaw_range", C.c_float),
        ("current_range", C.c_float), ("dr_scale_lo", C.c_float), ("dr_scale_hi", C.c_float),
        ("dr_buoy_range", C.c_float), ("dr_cob_range", C.c_float),
        ("hidden", C.c_int32), ("policy_out", C.c_int32), ("mlp_bf16", C.c_int32),
        ("has_value", C.c_int32), ("logstd_fixed", C.c_float * 8),
        ("logstd_min", C.c_float), ("logstd_max", C.c_float),
    ]


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        P = C.c_void_p
        _lib.oracle_model_size.restype = C.c_int
        _lib.oracle_philox.argtypes = [C.c_uint32, C.c_uint32, P, P]
        _lib.oracle_shac_window.argtypes = [C.POINTER(OracleModel), P, P, P, C.c_int, P, P, P, P,
                                            P, C.c_uint64, C.c_int, P, C.c_double, P, P]
        _lib.oracle_rbuf_indices.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint32, P]
        _lib.oracle_adjoint_window.argtypes = [C.POINTER(OracleModel), C.c_int, P, P, P, P, P,
                                               C.c_int, P, P, P, P, P, P, P]
        _lib.oracle_minibatch_perm.argtypes = [C.c_uint64, C.c_uint64, C.c_uint32, C.c_uint32,
                                               C.c_uint32, P]
        _lib.oracle_feistel.argtypes = [C.c_uint32, C.c_uint32, C.c_uint64, C.c_uint64, C.c_int]
        _lib.oracle_feistel.restype = C.c_uint32
        _lib.oracle_word_to_uniform.argtypes = [C.c_uint32]
        _lib.oracle_word_to_uniform.restype = C.c_float
        _lib.oracle_taylor_sin.argtypes = [C.c_float]
        _lib.oracle_taylor_sin.restype = C.c_float
        _lib.oracle_taylor_cos.argtypes = [C.c_float]
        _lib.oracle_taylor_cos.restype = C.c_float
        _lib.oracle_to_bf16.argtypes = [C.c_double]
        _lib.oracle_to_bf16.restype = C.c_float
        _lib.oracle_normals.argtypes = [C.c_uint32, C.c_uint32, C.c_uint64, P]
        _lib.oracle_reset.argtypes = [P, C.c_int, P, P, P, P, P]
        _lib.oracle_replay.argtypes = [P, C.c_int, C.c_int, P, P, P, P, P, C.c_int, P, P, P, P]
        _lib.oracle_rollout.argtypes = [P, C.c_int, P, P, C.c_int, P, P, P, P, P, C.c_uint64,
                                        C.c_int, P, P, P, P, P, P]
        _lib.oracle_mlp.argtypes = [P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int, P, P]
        _lib.oracle_policy_act.argtypes = [P, P, C.c_int, P, C.c_uint64, P, P, P, P]
        _lib.oracle_observe.argtypes = [P, P, P, P]
        _lib.oracle_reward.argtypes = [P, P, P, P]
        _lib.oracle_reward.restype = C.c_double
        _lib.oracle_allocate.argtypes = [P, P, P]
        _lib.oracle_nu_dot.argtypes = [P, P, P, P, P]
        _lib.oracle_integrate.argtypes = [P, C.c_int, P, P, P, C.c_double, C.c_int]
        assert _lib.oracle_model_size() == C.sizeof(OracleModel), "OracleModel layout mismatch"
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def model(w: dict) -> OracleModel:
    """OracleModel from a workload dict (paper_2512_13359_gb300.workloads)."""
    m = OracleModel()
    m.n_substeps = int(w["substeps"])
    m.episode_len = int(w["episode_len"])
    m.seed = int(w["seed"]) & 0xFFFFFFFF
    m.dr_enable = int(w["dr_enable"])
    m.dt = float(w["dt"])
    m.mass = float(w["mass"])
    m.inertia[:] = [float(x) for x in w["inertia"]]
    m.added_mass[:] = [float(x) for x in w["added_mass"]]
    m.damp_lin[:] = [float(x) for x in w["damp_lin"]]
    m.damp_quad[:] = [float(x) for x in w["damp_quad"]]
    m.gravity[:] = [float(x) for x in w["gravity"]]
    m.thrust_max = float(w["thrust_max"])
    m.alloc[:] = [float(x) for x in np.asarray(w["alloc"], dtype=np.float64).reshape(-1)]
    m.w_pos, m.w_att, m.w_act, m.w_vs = (float(w[k]) for k in ("w_pos", "w_att", "w_act", "w_vs"))
    for k in ("init_pos_range", "init_att_range", "goal_pos_range", "goal_yaw_range",
              "current_range", "dr_scale_lo", "dr_scale_hi", "dr_buoy_range", "dr_cob_range"):
        setattr(m, k, float(w[k]))
    m.hidden = int(w["hidden"])
    m.policy_out = int(w["policy_out"])
    m.mlp_bf16 = 1 if w["mlp"] == "bf16" else 0
    m.has_value = int(w["has_value"])
    m.logstd_fixed[:] = [float(x) for x in w["logstd_fixed"]]
    m.logstd_min = float(w["logstd_min"])
    m.logstd_max = float(w["logstd_max"])
    return m


class Batch:
    """SoA env batch held by the oracle: state[19][n], params[17][n] (float64),
    t_ep[n] (int32), episode[n] (uint32) for the listed env ids."""

    def __init__(self, env_ids):
        self.env_ids = np.ascontiguousarray(env_ids, dtype=np.uint32)
        n = len(self.env_ids)
        self.n = n
        self.state = np.zeros((19, n), dtype=np.float64)
        self.params = np.zeros((17, n), dtype=np.float64)
        self.t_ep = np.zeros(n, dtype=np.int32)
        self.episode = np.zeros(n, dtype=np.uint32)

    def copy(self):
        b = Batch(self.env_ids)
        b.state[:] = self.state
        b.params[:] = self.params
        b.t_ep[:] = self.t_ep
        b.episode[:] = self.episode
        return b


def reset(m: OracleModel, batch: Batch) -> Batch:
    lib().oracle_reset(C.byref(m), batch.n, _p(batch.env_ids), _p(batch.state),
                       _p(batch.params), _p(batch.t_ep), _p(batch.episode))
    return batch


def adjoint_window(m: OracleModel, batch: Batch, actions, coef, lam_T, dir_s0, dir_act):
    """J = sum_t coef[t] r_t + <lam_T, x_T> of an action-replay window from the
    batch's state (x = p, q, nu: 13 rows) and its directional derivative
    along (dir_s0 [13][n], dir_act [T][8][n]), by forward-mode dual numbers.
    The batch is not modified.  Returns (J[n], dJ[n])."""
    act = np.ascontiguousarray(actions, dtype=np.float64)
    T = act.shape[0]
    n = batch.n
    assert act.shape == (T, 8, n)
    coef = np.ascontiguousarray(coef, dtype=np.float64)
    assert coef.shape == (T,)
    lam = None if lam_T is None else np.ascontiguousarray(lam_T, dtype=np.float64)
    ds0 = np.ascontiguousarray(dir_s0, dtype=np.float64)
    da = np.ascontiguousarray(dir_act, dtype=np.float64)
    assert ds0.shape == (13, n) and da.shape == act.shape
    J = np.zeros(n)
    dJ = np.zeros(n)
    lib().oracle_adjoint_window(C.byref(m), n, _p(batch.env_ids), _p(batch.state),
                                _p(batch.params), _p(batch.t_ep), _p(batch.episode), T, _p(act),
                                _p(coef), _p(lam), _p(ds0), _p(da), _p(J), _p(dJ))
    return J, dJ


def shac_window(m: OracleModel, batch: Batch, pol_w, dpol, val_w, t_g0: int, T: int, coef,
                coef_V: float):
    """SHAC window objective per env in closed loop (policy head 16, noise
    of global steps t_g0 ..) and its directional derivative along the
    policy-weight direction dpol (or None).  The batch is not modified.
    Returns (J[n], dJ[n])."""
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    dp = None if dpol is None else np.ascontiguousarray(dpol, dtype=np.float64)
    vw = None if val_w is None else np.ascontiguousarray(val_w, dtype=np.float32)
    coef = np.ascontiguousarray(coef, dtype=np.float64)
    assert coef.shape == (T,) and m.policy_out == 16
    n = batch.n
    J = np.zeros(n)
    dJ = np.zeros(n)
    lib().oracle_shac_window(C.byref(m), _p(pw), _p(dp), _p(vw), n, _p(batch.env_ids),
                             _p(batch.state), _p(batch.params), _p(batch.t_ep), _p(batch.episode),
                             t_g0, T, _p(coef), float(coef_V), _p(J), _p(dJ))
    return J, dJ


def replay(m: OracleModel, batch: Batch, actions: np.ndarray, precision: str = "f64",
           trace: bool = False):
    """Action replay over T steps; actions[T][8][n] float32.  Mutates batch.
    Returns (rew[T][n], done[T][n], trace[T][19][n] or None)."""
    T = actions.shape[0]
    n = batch.n
    assert actions.shape == (T, 8, n)
    act = np.ascontiguousarray(actions, dtype=np.float32)
    rew = np.zeros((T, n), dtype=np.float64)
    done = np.zeros((T, n), dtype=np.uint8)
    tr = np.zeros((T, 19, n), dtype=np.float64) if trace else None
    lib().oracle_replay(C.byref(m), 1 if precision == "f32" else 0, n, _p(batch.env_ids),
                        _p(batch.state), _p(batch.params), _p(batch.t_ep), _p(batch.episode),
                        T, _p(act), _p(rew), _p(done), _p(tr))
    return rew, done, tr


def rollout(m: OracleModel, batch: Batch, pol_w: np.ndarray, val_w, t_g0: int, T: int,
            precision: str = "f64", want=("obs", "act", "logp", "value", "rew", "done")):
    """Closed-loop rollout over T steps.  Mutates batch.  Returns a dict of
    SoA arrays obs[T][18][n], act[T][8][n], logp[T][n], value[T][n],
    rew[T][n], done[T][n] (those listed in `want`)."""
    n = batch.n
    out = {}
    shapes = dict(obs=(T, 18, n), act=(T, 8, n), logp=(T, n), value=(T, n), rew=(T, n))
    for k, s in shapes.items():
        out[k] = np.zeros(s, dtype=np.float64) if k in want else None
    if "value" in want and not m.has_value:
        out["value"] = None
    out["done"] = np.zeros((T, n), dtype=np.uint8)
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    vw = None if val_w is None else np.ascontiguousarray(val_w, dtype=np.float32)
    lib().oracle_rollout(C.byref(m), 1 if precision == "f32" else 0, _p(pw), _p(vw), n,
                         _p(batch.env_ids), _p(batch.state), _p(batch.params), _p(batch.t_ep),
                         _p(batch.episode), int(t_g0), T, _p(out["obs"]), _p(out["act"]),
                         _p(out["logp"]), _p(out["value"]), _p(out["rew"]), _p(out["done"]))
    return {k: v for k, v in out.items() if v is not None}


def mlp(weights: np.ndarray, in_dim: int, hidden: int, out_dim: int, bf16: bool,
        x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    n = x.shape[0]
    out = np.zeros((n, out_dim), dtype=np.float64)
    w = np.ascontiguousarray(weights, dtype=np.float32)
    lib().oracle_mlp(_p(w), in_dim, hidden, out_dim, 1 if bf16 else 0, n, _p(x), _p(out))
    return out


def policy_act(m: OracleModel, pol_w, env_ids, t_g: int, obs: np.ndarray, with_mu=False):
    """One policy draw per row of obs[n][18] (env ids env_ids, global step
    t_g): the network head, the clamped (or fixed) log-std, the step's
    normals, a = mu + sigma eps and log pi(a).  Returns (act[n][8], logp[n])
    and, with with_mu, the mean mu[n][8] as a third array."""
    ids = np.ascontiguousarray(env_ids, dtype=np.uint32)
    x = np.ascontiguousarray(obs, dtype=np.float64)
    n = len(ids)
    assert x.shape == (n, 18)
    act = np.zeros((n, 8))
    logp = np.zeros(n)
    mu = np.zeros((n, 8)) if with_mu else None
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    lib().oracle_policy_act(C.byref(m), _p(pw), n, _p(ids), int(t_g), _p(x), _p(act), _p(logp),
                            _p(mu))
    return (act, logp, mu) if with_mu else (act, logp)


def philox(key0: int, key1: int, ctr) -> np.ndarray:
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_philox(key0 & 0xFFFFFFFF, key1 & 0xFFFFFFFF, _p(c), _p(out))
    return out


def minibatch_perm(seed: int, epoch: int, m: int, start: int, count: int) -> np.ndarray:
    """Positions start .. start+count-1 of the learner's epoch permutation of [0, m)."""
    out = np.zeros(count, dtype=np.uint32)
    lib().oracle_minibatch_perm(seed, epoch, m, start, count, _p(out))
    return out


def rbuf_indices(seed: int, draw: int, size: int, count: int) -> np.ndarray:
    """Replay-buffer sample indices of draw `draw` (see oracle_rbuf_indices)."""
    out = np.zeros(count, dtype=np.uint32)
    lib().oracle_rbuf_indices(seed, draw, size, count, _p(out))
    return out


def feistel(x: int, m: int, seed: int, epoch: int, inverse: bool = False) -> int:
    return int(lib().oracle_feistel(x, m, seed, epoch, 1 if inverse else 0))


def normals(env_id: int, seed: int, t_g: int) -> np.ndarray:
    out = np.zeros(8, dtype=np.float64)
    lib().oracle_normals(env_id, seed, t_g, _p(out))
    return out


def single_env(state: dict, params: dict):
    """19- and 17-row single-env SoA vectors from field dicts (missing = 0,
    scales default 1, quaternions default identity)."""
    st = np.zeros(19)
    pr = np.zeros(17)
    st[3] = 1.0
    pr[3] = 1.0
    pr[7] = pr[8] = pr[9] = 1.0
    for k, v in state.items():
        idx = dict(p=0, q=3, nu=7, nu_prev=13)[k]
        st[idx:idx + len(v)] = v
    for k, v in params.items():
        idx = dict(p_d=0, q_d=3, s_m=7, s_a=8, s_d=9, dB=10, r_b=11, V_c=14)[k]
        v = np.atleast_1d(v)
        pr[idx:idx + len(v)] = v
    return st, pr


def observe(st, pr):
    obs = np.zeros(18)
    th = np.zeros(1)
    lib().oracle_observe(_p(np.ascontiguousarray(st, dtype=np.float64)),
                         _p(np.ascontiguousarray(pr, dtype=np.float64)), _p(obs), _p(th))
    return obs, float(th[0])


def reward(m, st, pr, a_c):
    return lib().oracle_reward(C.byref(m), _p(np.ascontiguousarray(st, dtype=np.float64)),
                               _p(np.ascontiguousarray(pr, dtype=np.float64)),
                               _p(np.ascontiguousarray(a_c, dtype=np.float64)))


def allocate(m, a):
    tau = np.zeros(6)
    lib().oracle_allocate(C.byref(m), _p(np.ascontiguousarray(a, dtype=np.float64)), _p(tau))
    return tau


def nu_dot(m, st, pr, tau):
    out = np.zeros(6)
    lib().oracle_nu_dot(C.byref(m), _p(np.ascontiguousarray(st, dtype=np.float64)),
                        _p(np.ascontiguousarray(pr, dtype=np.float64)),
                        _p(np.ascontiguousarray(tau, dtype=np.float64)), _p(out))
    return out


def integrate(m, st, pr, tau, h, n_steps, method="euler"):
    """Integrate one env's physics; returns the new 19-row state vector."""
    s = np.ascontiguousarray(st, dtype=np.float64).copy()
    lib().oracle_integrate(C.byref(m), 0 if method == "euler" else 1, _p(s),
                           _p(np.ascontiguousarray(pr, dtype=np.float64)),
                           _p(np.ascontiguousarray(tau, dtype=np.float64)), float(h),
                           int(n_steps))
    return s


# ---------------------------------------------------------------------------
# The paper's own environment (§IV-B; see PaperModel in auv_oracle.cpp)
# ---------------------------------------------------------------------------
PAPER_OBS, PAPER_ACT, PAPER_HIST = 12, 6, 8
PAPER_STATE, PAPER_PARAM = 13 + 6 * PAPER_HIST, 8


class PaperModel(C.Structure):
    _fields_ = [
        ("n_substeps", C.c_int32), ("episode_len", C.c_int32), ("seed", C.c_uint32),
        ("dr_enable", C.c_int32), ("mavg_len", C.c_int32), ("pad0", C.c_int32),
        ("dt", C.c_double), ("mass", C.c_double), ("inertia", C.c_double * 3),
        ("f_max", C.c_double), ("tau_max", C.c_double), ("rho", C.c_double),
        ("visc", C.c_double), ("g_eff", C.c_double),
        ("w_pos", C.c_double), ("w_axes", C.c_double * 3), ("w_att", C.c_double),
        ("w_act", C.c_double), ("w_vel", C.c_double), ("w_mavg", C.c_double),
        ("goal_pos_range", C.c_float), ("goal_att_range", C.c_float),
        ("init_pos_range", C.c_float), ("init_att_range", C.c_float),
        ("dr_gravity_range", C.c_float),
        ("hidden", C.c_int32), ("policy_out", C.c_int32), ("mlp_bf16", C.c_int32),
        ("has_value", C.c_int32), ("logstd_fixed", C.c_float * 6),
        ("logstd_min", C.c_float), ("logstd_max", C.c_float),
    ]


def _paper_lib():
    L = lib()
    if not getattr(L, "_paper_ready", False):
        P = C.c_void_p
        L.oracle_paper_model_size.restype = C.c_int
        L.oracle_paper_reset.argtypes = [P, C.c_int, P, P, P, P, P]
        L.oracle_paper_replay.argtypes = [P, C.c_int, C.c_int, P, P, P, P, P, C.c_int, P, P, P,
                                          P]
        L.oracle_paper_rollout.argtypes = [P, C.c_int, P, P, C.c_int, P, P, P, P, P,
                                           C.c_uint64, C.c_int, P, P, P, P, P, P]
        L.oracle_paper_observe.argtypes = [P, P, P]
        L.oracle_paper_policy_act.argtypes = [P, P, C.c_int, P, C.c_uint64, P, P, P, P]
        L.oracle_paper_reward.argtypes = [P, P, P, P]
        L.oracle_paper_reward.restype = C.c_double
        L.oracle_paper_wrench.argtypes = [P, P, P, P]
        L.oracle_paper_box.argtypes = [P, P]
        L.oracle_paper_nu_dot.argtypes = [P, P, P, P, P]
        L.oracle_paper_integrate.argtypes = [P, C.c_int, P, P, P, C.c_double, C.c_int]
        L.oracle_paper_adjoint_window.argtypes = [P, C.c_int, P, P, P, P, P, C.c_int, P, P, P,
                                                  P, P, P, P]
        L.oracle_paper_shac_window.argtypes = [P, P, P, P, C.c_int, P, P, P, P, P, C.c_uint64,
                                               C.c_int, P, C.c_double, P, P]
        assert L.oracle_paper_model_size() == C.sizeof(PaperModel), "PaperModel layout mismatch"
        L._paper_ready = True
    return L


def paper_model(w: dict) -> PaperModel:
    """PaperModel from a paper-model workload dict."""
    m = PaperModel()
    m.n_substeps = int(w["substeps"])
    m.episode_len = int(w["episode_len"])
    m.seed = int(w["seed"]) & 0xFFFFFFFF
    m.dr_enable = int(w["dr_enable"])
    m.mavg_len = int(w["mavg_len"])
    m.dt = float(w["dt"])
    m.mass = float(w["mass"])
    m.inertia[:] = [float(x) for x in w["inertia"]]
    m.f_max, m.tau_max = float(w["f_max"]), float(w["tau_max"])
    m.rho, m.visc = float(w["fluid_density"]), float(w["fluid_viscosity"])
    m.g_eff = float(w["g_eff"])
    m.w_pos = float(w["w_pos"])
    m.w_axes[:] = [float(x) for x in w["w_axes"]]
    m.w_att, m.w_act, m.w_vel, m.w_mavg = (float(w[k]) for k in ("w_att", "w_act", "w_vel",
                                                                   "w_mavg"))
    for k in ("goal_pos_range", "goal_att_range", "init_pos_range", "init_att_range",
              "dr_gravity_range"):
        setattr(m, k, float(w[k]))
    m.hidden = int(w["hidden"])
    m.policy_out = int(w["policy_out"])
    m.mlp_bf16 = 1 if w["mlp"] == "bf16" else 0
    m.has_value = int(w["has_value"])
    m.logstd_fixed[:] = [float(x) for x in w["logstd_fixed"][:6]]
    m.logstd_min = float(w["logstd_min"])
    m.logstd_max = float(w["logstd_max"])
    return m


class PaperBatch(Batch):
    """SoA batch of the paper model: state[61][n] (p q nu, action history
    [8][6]), params[8][n] (p_d q_d g_eff), t_ep, episode."""

    def __init__(self, env_ids):
        self.env_ids = np.ascontiguousarray(env_ids, dtype=np.uint32)
        n = len(self.env_ids)
        self.n = n
        self.state = np.zeros((PAPER_STATE, n), dtype=np.float64)
        self.params = np.zeros((PAPER_PARAM, n), dtype=np.float64)
        self.t_ep = np.zeros(n, dtype=np.int32)
        self.episode = np.zeros(n, dtype=np.uint32)

    def copy(self):
        b = PaperBatch(self.env_ids)
        b.state[:] = self.state
        b.params[:] = self.params
        b.t_ep[:] = self.t_ep
        b.episode[:] = self.episode
        return b


def paper_reset(m: PaperModel, batch: PaperBatch) -> PaperBatch:
    _paper_lib().oracle_paper_reset(C.byref(m), batch.n, _p(batch.env_ids), _p(batch.state),
                                    _p(batch.params), _p(batch.t_ep), _p(batch.episode))
    return batch


def paper_replay(m: PaperModel, batch: PaperBatch, actions: np.ndarray, precision="f64",
                 trace=False):
    """actions[T][6][n]; returns (rew[T][n], done[T][n], trace[T][61][n] or None)."""
    T, n = actions.shape[0], batch.n
    assert actions.shape == (T, PAPER_ACT, n)
    act = np.ascontiguousarray(actions, dtype=np.float32)
    rew = np.zeros((T, n))
    done = np.zeros((T, n), dtype=np.uint8)
    tr = np.zeros((T, PAPER_STATE, n)) if trace else None
    _paper_lib().oracle_paper_replay(C.byref(m), 1 if precision == "f32" else 0, n,
                                     _p(batch.env_ids), _p(batch.state), _p(batch.params),
                                     _p(batch.t_ep), _p(batch.episode), T, _p(act), _p(rew),
                                     _p(done), _p(tr))
    return rew, done, tr


def paper_adjoint_window(m: PaperModel, batch: PaperBatch, actions, coef, lam_T, dir_s0,
                         dir_act):
    """The paper model's window objective (state rows 0..60: p, q, nu and
    the action history) and its directional derivative, in dual numbers.
    Returns (J[n], dJ[n]); the batch is not modified."""
    act = np.ascontiguousarray(actions, dtype=np.float64)
    T, n = act.shape[0], batch.n
    assert act.shape == (T, PAPER_ACT, n)
    coef = np.ascontiguousarray(coef, dtype=np.float64)
    lam = None if lam_T is None else np.ascontiguousarray(lam_T, dtype=np.float64)
    ds0 = np.ascontiguousarray(dir_s0, dtype=np.float64)
    da = np.ascontiguousarray(dir_act, dtype=np.float64)
    assert ds0.shape == (PAPER_STATE, n) and da.shape == act.shape
    J = np.zeros(n)
    dJ = np.zeros(n)
    _paper_lib().oracle_paper_adjoint_window(C.byref(m), n, _p(batch.env_ids), _p(batch.state),
                                             _p(batch.params), _p(batch.t_ep),
                                             _p(batch.episode), T, _p(act), _p(coef), _p(lam),
                                             _p(ds0), _p(da), _p(J), _p(dJ))
    return J, dJ


def paper_shac_window(m: PaperModel, batch: PaperBatch, pol_w, dpol, val_w, t_g0: int, T: int,
                      coef, coef_V: float):
    """SHAC's closed-loop window on the paper model (policy head 12) and its
    derivative along the policy-weight direction dpol (or None)."""
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    dp = None if dpol is None else np.ascontiguousarray(dpol, dtype=np.float64)
    vw = None if val_w is None else np.ascontiguousarray(val_w, dtype=np.float32)
    coef = np.ascontiguousarray(coef, dtype=np.float64)
    assert coef.shape == (T,) and m.policy_out == 12
    n = batch.n
    J = np.zeros(n)
    dJ = np.zeros(n)
    _paper_lib().oracle_paper_shac_window(C.byref(m), _p(pw), _p(dp), _p(vw), n,
                                          _p(batch.env_ids), _p(batch.state), _p(batch.params),
                                          _p(batch.t_ep), _p(batch.episode), t_g0, T, _p(coef),
                                          float(coef_V), _p(J), _p(dJ))
    return J, dJ


def paper_rollout(m: PaperModel, batch: PaperBatch, pol_w, val_w, t_g0: int, T: int,
                  precision="f64", want=("obs", "act", "logp", "value", "rew", "done")):
    """obs[T][12][n], act[T][6][n], logp, value, rew, done (those in `want`)."""
    n = batch.n
    out = {}
    shapes = dict(obs=(T, PAPER_OBS, n), act=(T, PAPER_ACT, n), logp=(T, n), value=(T, n),
                  rew=(T, n))
    for k, s in shapes.items():
        out[k] = np.zeros(s) if k in want else None
    if "value" in want and not m.has_value:
        out["value"] = None
    out["done"] = np.zeros((T, n), dtype=np.uint8)
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    vw = None if val_w is None else np.ascontiguousarray(val_w, dtype=np.float32)
    _paper_lib().oracle_paper_rollout(C.byref(m), 1 if precision == "f32" else 0, _p(pw),
                                      _p(vw), n, _p(batch.env_ids), _p(batch.state),
                                      _p(batch.params), _p(batch.t_ep), _p(batch.episode),
                                      int(t_g0), T, _p(out["obs"]), _p(out["act"]),
                                      _p(out["logp"]), _p(out["value"]), _p(out["rew"]),
                                      _p(out["done"]))
    return {k: v for k, v in out.items() if v is not None}


def paper_policy_act(m: PaperModel, pol_w, env_ids, t_g: int, obs: np.ndarray, with_mu=False):
    """The paper model's policy draw per row of obs[n][12]: (act[n][6],
    logp[n]) and, with with_mu, the mean mu[n][6]."""
    ids = np.ascontiguousarray(env_ids, dtype=np.uint32)
    x = np.ascontiguousarray(obs, dtype=np.float64)
    n = len(ids)
    assert x.shape == (n, PAPER_OBS)
    act = np.zeros((n, PAPER_ACT))
    logp = np.zeros(n)
    mu = np.zeros((n, PAPER_ACT)) if with_mu else None
    pw = np.ascontiguousarray(pol_w, dtype=np.float32)
    _paper_lib().oracle_paper_policy_act(C.byref(m), _p(pw), n, _p(ids), int(t_g), _p(x),
                                         _p(act), _p(logp), _p(mu))
    return (act, logp, mu) if with_mu else (act, logp)


def paper_single_env(state: dict, params: dict):
    """61- and 8-row single-env vectors from field dicts (missing = 0,
    quaternions default identity).  State keys p, q, nu, hist ([8][6]);
    param keys p_d, q_d, g_eff."""
    st = np.zeros(PAPER_STATE)
    pr = np.zeros(PAPER_PARAM)
    st[3] = 1.0
    pr[3] = 1.0
    for k, v in state.items():
        if k == "hist":
            st[13:13 + 6 * PAPER_HIST] = np.asarray(v, dtype=np.float64).reshape(-1)
            continue
        idx = dict(p=0, q=3, nu=7)[k]
        st[idx:idx + len(v)] = v
    for k, v in params.items():
        idx = dict(p_d=0, q_d=3, g_eff=7)[k]
        v = np.atleast_1d(v)
        pr[idx:idx + len(v)] = v
    return st, pr


def _d(a):
    return _p(np.ascontiguousarray(a, dtype=np.float64))


def paper_observe(st, pr):
    obs = np.zeros(PAPER_OBS)
    _paper_lib().oracle_paper_observe(_d(st), _d(pr), _p(obs))
    return obs


def paper_reward(m, st, pr, a_c):
    return _paper_lib().oracle_paper_reward(C.byref(m), _d(st), _d(pr), _d(a_c))


def paper_wrench(m, a):
    a_c, tau = np.zeros(PAPER_ACT), np.zeros(6)
    _paper_lib().oracle_paper_wrench(C.byref(m), _d(a), _p(a_c), _p(tau))
    return a_c, tau


def paper_box(m):
    b = np.zeros(3)
    _paper_lib().oracle_paper_box(C.byref(m), _p(b))
    return b


def paper_nu_dot(m, st, pr, tau):
    out = np.zeros(6)
    _paper_lib().oracle_paper_nu_dot(C.byref(m), _d(st), _d(pr), _d(tau), _p(out))
    return out


def paper_integrate(m, st, pr, tau, h, n_steps, method="euler"):
    s = np.ascontiguousarray(st, dtype=np.float64).copy()
    _paper_lib().oracle_paper_integrate(C.byref(m), 0 if method == "euler" else 1, _p(s),
                                        _d(pr), _d(tau), float(h), int(n_steps))
    return s
