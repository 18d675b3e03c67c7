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
"""
from __future__ import annotations

import copy
import math

import numpy as np

OBS_DIM = 18
ACT_DIM = 8
STATE_FIELDS = 19   # p(3) q(4) nu(6) nu_prev(6)
PARAM_FIELDS = 17   # p_d(3) q_d(4) s_m s_a s_d dB r_b(3) V_c(3)

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
SWEEP_SIZES = (1024, 4096, 16384, 65536, 262144, 1048576)


def workload(name: str, **overrides) -> dict:
    """A deep copy of a preset with overrides, vehicle constants merged in."""
    w = copy.deepcopy(WORKLOADS[name])
    w.update(copy.deepcopy(VEHICLE))
    w["alloc"] = allocation_matrix()
    w["name"] = name
    w.update(overrides)
    return w


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
    return mlp_weights(w["weight_seed"], OBS_DIM, w["hidden"], w["policy_out"], 0, bias_std)


def value_weights(w: dict, bias_std: float = 0.0) -> np.ndarray:
    return mlp_weights(w["weight_seed"], OBS_DIM, w["hidden"], 1, 1, bias_std)


def replay_actions(seed: int, T: int, n: int, scale: float = 0.7) -> np.ndarray:
    """Normalised thruster commands [T][8][n] (float32) for action-replay runs:
    N(0, scale^2), so a share of them saturate at the +-1 clip."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 7]))
    return (rng.standard_normal((T, ACT_DIM, n)) * scale).astype(np.float32)


def random_observations(seed: int, n: int) -> np.ndarray:
    """Observation-shaped inputs [n][18] for network-only checks: position
    errors ~ +-2 m, rotation-matrix entries in [-1, 1], velocities ~ +-1."""
    rng = np.random.Generator(np.random.Philox(key=[seed, 11]))
    x = np.empty((n, OBS_DIM), dtype=np.float64)
    x[:, 0:3] = rng.uniform(-2, 2, (n, 3))
    x[:, 3:12] = rng.uniform(-1, 1, (n, 9))
    x[:, 12:18] = rng.uniform(-1, 1, (n, 6))
    return x.astype(np.float32)
