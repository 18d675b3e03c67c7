"""Seeded synthetic inputs for the batched AUV rollout.

This module is the ONE place shared by the CUDA path, the CPU oracle, the
tests and the benchmark.  It holds workload presets (sizes, vehicle constants,
ranges), the thruster geometry and seeded generators for network weights and
replay actions.  It contains none of the method's arithmetic: no dynamics, no
observation, no reward, no random stream of the method itself (those random
numbers are drawn inside each implementation from the counter-based Philox
definition).

The paper (arXiv 2512.13359) trains on fully synthetic episodes: random
references and initial states per episode (§V-A1) and per-env randomised
parameters (§IV-C).  It publishes no vehicle constants; the presets below fix
them (BlueROV2-Heavy-sized rigid body with diagonal added mass and linear plus
quadratic damping, 8 thrusters) and the sizes of the five workloads.

Two environment models exist (preset key "model"): "fossen", the
thruster-level Fossen model with added mass, currents and domain-randomised
parameters (18-float observation, 8 thruster commands), and "paper", the
paper's own environment (§IV-B): a 6-D body-wrench action scaled by F_max and
tau_max (Eq. 1), a free rigid body under the inertia-box fluid model with an
effective gravity randomised per episode (§IV-C), a 12-float axis-angle
observation and the five-term reward of Eqs. (2)-(7).
"""
from __future__ import annotations

import copy
import math

import numpy as np

OBS_DIM = 18
ACT_DIM = 8
STATE_FIELDS = 19   # p(3) q(4) nu(6) nu_prev(6)
PARAM_FIELDS = 17   # p_d(3) q_d(4) s_m s_a s_d dB r_b(3) V_c(3)

# The paper model: 12-float observation, 6-D wrench action; state p q nu and
# an 8-slot history of clipped actions; parameters p_d q_d g_eff.
PAPER_OBS_DIM = 12
PAPER_ACT_DIM = 6
PAPER_HIST = 8
PAPER_STATE_FIELDS = 13 + 6 * PAPER_HIST
PAPER_PARAM_FIELDS = 8

# Names of the SoA rows, for readable tests and snapshots.
STATE_NAMES = (["p_x", "p_y", "p_z", "q_w", "q_x", "q_y", "q_z"]
               + [f"nu_{k}" for k in range(6)] + [f"nu_prev_{k}" for k in range(6)])
PARAM_NAMES = (["pd_x", "pd_y", "pd_z", "qd_w", "qd_x", "qd_y", "qd_z",
                "s_m", "s_a", "s_d", "dB", "rb_x", "rb_y", "rb_z",
                "Vc_x", "Vc_y", "Vc_z"])


def thruster_geometry():
    """Positions r_i and unit directions d_i (body frame, x fwd, y left, z up)
    of an 8-thruster vectored layout: four horizontal thrusters at 45 degrees
    and four vertical thrusters."""
    s = 1.0 / math.sqrt(2.0)
    pos = [(0.15, 0.10, 0.0), (0.15, -0.10, 0.0), (-0.15, 0.10, 0.0), (-0.15, -0.10, 0.0),
           (0.12, 0.22, 0.0), (0.12, -0.22, 0.0), (-0.12, 0.22, 0.0), (-0.12, -0.22, 0.0)]
    dirs = [(s, -s, 0.0), (s, s, 0.0), (s, s, 0.0), (s, -s, 0.0),
            (0.0, 0.0, 1.0), (0.0, 0.0, 1.0), (0.0, 0.0, 1.0), (0.0, 0.0, 1.0)]
    return np.array(pos, dtype=np.float64), np.array(dirs, dtype=np.float64)


def allocation_matrix():
    """6x8 thruster allocation B: column i = [d_i; r_i x d_i] (force and
    moment per newton of thrust).  The rollout takes B as an input."""
    pos, dirs = thruster_geometry()
    B = np.zeros((6, 8), dtype=np.float64)
    for i in range(8):
        B[:3, i] = dirs[i]
        B[3:, i] = np.cross(pos[i], dirs[i])
    return B


VEHICLE = dict(
    mass=11.5,
    inertia=(0.16, 0.16, 0.16),
    added_mass=(5.5, 12.7, 14.6, 0.12, 0.12, 0.12),
    damp_lin=(4.0, 6.0, 5.0, 0.07, 0.07, 0.07),
    damp_quad=(18.0, 21.0, 37.0, 1.5, 1.5, 1.5),
    gravity=(0.0, 0.0, -9.81),
    thrust_max=40.0,
)

_BASE = dict(
    n_envs=64, steps=200, substeps=1, dt=0.02, episode_len=500, seed=0,
    weight_seed=0,
    init_pos_range=0.5, init_att_range=0.3, goal_pos_range=1.0, goal_yaw_range=math.pi,
    current_range=0.0, dr_enable=0, dr_scale_lo=0.8, dr_scale_hi=1.2,
    dr_buoy_range=2.0, dr_cob_range=0.01,
    w_pos=1.0, w_att=0.5, w_act=0.01, w_vs=0.0,
    hidden=64, policy_out=8, mlp="fp32", has_value=0,
    logstd_fixed=(0.0,) * 8, logstd_min=-5.0, logstd_max=2.0,
    trajectory="reward_done",
)

# Paper-model constants (§IV-B names the quantities, not their values): the
# same rigid body without added mass; water; a neutrally buoyant nominal
# vehicle whose effective gravity is randomised by +-0.2 m/s^2; goals within
# +-2 m and +-60 degrees as in §V-A1; 512-step episodes.
PAPER_MODEL = dict(
    model="paper", f_max=40.0, tau_max=10.0, fluid_density=1000.0, fluid_viscosity=0.001,
    g_eff=0.0, dr_gravity_range=0.2, w_axes=(1.0, 1.0, 1.0), w_pos=1.0, w_att=0.5,
    w_act=0.01, w_vel=0.05, w_mavg=0.1, mavg_len=4, goal_pos_range=2.0,
    goal_att_range=math.pi / 3, init_pos_range=0.0, init_att_range=0.0, episode_len=512,
    policy_out=6, logstd_fixed=(0.0,) * 6,
)

# The five workloads.  "tiny" is the case the oracle finishes in seconds.
WORKLOADS = {
    "tiny_64": dict(_BASE),
    "fp32_4096": dict(_BASE, n_envs=4096, steps=1000, substeps=4, hidden=256),
    "dr_16384": dict(_BASE, n_envs=16384, steps=1000, substeps=4, hidden=256,
                     dr_enable=1, current_range=0.3),
    "ppo_65536": dict(_BASE, n_envs=65536, steps=128, substeps=4, hidden=256,
                      dr_enable=1, current_range=0.3, policy_out=16, mlp="bf16",
                      has_value=1, trajectory="full"),
}
WORKLOADS["sweep"] = dict(WORKLOADS["ppo_65536"], steps=256)
# The paper's own environment: a small oracle-sized case and the paper's
# largest setting (4,096 envs, one 512-step episode), with the 65,536-env
# workload's network shapes (mean and log-std head, value network, bf16).
WORKLOADS["paper_tiny"] = dict(_BASE, **PAPER_MODEL)
WORKLOADS["paper_4096"] = dict(_BASE, **PAPER_MODEL, n_envs=4096, steps=512, substeps=4,
                               hidden=256, dr_enable=1, mlp="bf16", has_value=1,
                               trajectory="full")
WORKLOADS["paper_4096"]["policy_out"] = 12
SWEEP_SIZES = (1024, 4096, 16384, 65536, 262144, 1048576)


def workload(name: str, **overrides) -> dict:
    """A deep copy of a preset with overrides, vehicle constants merged in."""
    w = dict(model="fossen")
    w.update(copy.deepcopy(WORKLOADS[name]))
    w.update(copy.deepcopy(VEHICLE))
    w["alloc"] = allocation_matrix()
    w["name"] = name
    w.update(overrides)
    return w


def is_paper(w: dict) -> bool:
    return w.get("model", "fossen") == "paper"


def obs_dim(w: dict) -> int:
    return PAPER_OBS_DIM if is_paper(w) else OBS_DIM


def act_dim(w: dict) -> int:
    return PAPER_ACT_DIM if is_paper(w) else ACT_DIM


def state_fields(w: dict) -> int:
    return PAPER_STATE_FIELDS if is_paper(w) else STATE_FIELDS


def param_fields(w: dict) -> int:
    return PAPER_PARAM_FIELDS if is_paper(w) else PARAM_FIELDS


def mlp_shapes(in_dim: int, hidden: int, out_dim: int):
    """(name, shape) of the flat [W1 | b1 | W2 | b2 | W3 | b3] layout, rows = out."""
    return [("W1", (hidden, in_dim)), ("b1", (hidden,)), ("W2", (hidden, hidden)),
            ("b2", (hidden,)), ("W3", (out_dim, hidden)), ("b3", (out_dim,))]


def mlp_param_count(in_dim: int, hidden: int, out_dim: int) -> int:
    return sum(int(np.prod(s)) for _, s in mlp_shapes(in_dim, hidden, out_dim))


def mlp_weights(seed: int, in_dim: int, hidden: int, out_dim: int, stream: int = 0,
                bias_std: float = 0.0) -> np.ndarray:
    """Flat float32 weights, W ~ N(0, 1/fan_in), biases 0 (or N(0, bias_std^2)
    for tests that need the bias path exercised).  numpy's Philox bit generator
    keyed by (seed, stream)."""
    rng = np.random.Generator(np.random.Philox(key=[seed, stream]))
    parts = []
    for name, shape in mlp_shapes(in_dim, hidden, out_dim):
        if name.startswith("W"):
            fan_in = shape[1]
            parts.append(rng.standard_normal(shape) / math.sqrt(fan_in))
        else:
            parts.append(rng.standard_normal(shape) * bias_std if bias_std else np.zeros(shape))
    return np.concatenate([p.reshape(-1) for p in parts]).astype(np.float32)


def policy_weights(w: dict, bias_std: float = 0.0) -> np.ndarray:
    return mlp_weights(w["weight_seed"], obs_dim(w), w["hidden"], w["policy_out"], 0, bias_std)


def value_weights(w: dict, bias_std: float = 0.0) -> np.ndarray:
    return mlp_weights(w["weight_seed"], obs_dim(w), w["hidden"], 1, 1, bias_std)


def replay_actions(seed: int, T: int, n: int, scale: float = 0.7,
                   act: int = ACT_DIM) -> np.ndarray:
    """Normalised commands [T][act][n] (float32) for action-replay runs:
    N(0, scale^2), so a share of them saturate at the +-1 clip."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 7]))
    return (rng.standard_normal((T, act, n)) * scale).astype(np.float32)


def random_observations(seed: int, n: int, dim: int = OBS_DIM) -> np.ndarray:
    """Observation-shaped inputs [n][dim] for network-only checks: position
    errors ~ +-2 m, then attitude entries in [-1, 1] (rotation matrix, 18
    floats) or +-pi/2 (axis-angle, 12 floats), velocities ~ +-1."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 11]))
    x = np.empty((n, dim), dtype=np.float64)
    x[:, 0:3] = rng.uniform(-2, 2, (n, 3))
    if dim == OBS_DIM:
        x[:, 3:12] = rng.uniform(-1, 1, (n, 9))
    else:
        x[:, 3:6] = rng.uniform(-1.5, 1.5, (n, 3))
    x[:, dim - 6:dim] = rng.uniform(-1, 1, (n, 6))
    return x.astype(np.float32)
