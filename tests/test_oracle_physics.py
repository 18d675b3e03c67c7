"""Pins for the oracle's dynamics against what physics fixes independently of
the code: rest equilibrium, unit quaternion, energy decay, rotation
invariance, first-order convergence to an RK4 brute force, 1-DOF closed forms
(Bernoulli decay, terminal velocity, buoyancy acceleration, pendulum period,
constant spin), Kirchhoff's impulse invariants of a body in ideal fluid, the
Munk moment, and Galilean invariance under a uniform current."""
import math

import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W

NO_DAMP = dict(damp_lin=(0.0,) * 6, damp_quad=(0.0,) * 6)


def _model(oracle, **over):
    return oracle.model(W.workload("tiny_64", **over))


def _quat_mul(a, b):
    w1, x1, y1, z1 = a
    w2, x2, y2, z2 = b
    return np.array([w1 * w2 - x1 * x2 - y1 * y2 - z1 * z2,
                     w1 * x2 + x1 * w2 + y1 * z2 - z1 * y2,
                     w1 * y2 - x1 * z2 + y1 * w2 + z1 * x2,
                     w1 * z2 + x1 * y2 - y1 * x2 + z1 * w2])


def _rot(q):
    from scipy.spatial.transform import Rotation
    return Rotation.from_quat([q[1], q[2], q[3], q[0]]).as_matrix()


def _random_quat(rng):
    q = rng.standard_normal(4)
    return q / np.linalg.norm(q)


def _mass_diag(w, s_m=1.0, s_a=1.0):
    return np.array([s_m * w["mass"]] * 3 + [s_m * x for x in w["inertia"]]) + \
        s_a * np.array(w["added_mass"])


# ----------------------------------------------------------------------------
# Invariants
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("precision", ["f64", "f32"])
def test_neutral_vehicle_at_rest_stays_at_rest(oracle, precision):
    """Neutral buoyancy (dB = 0, r_b = 0), no current, zero thrust: velocity
    stays exactly zero, position exactly unchanged, and the attitude is the
    initial one (renormalised once: the float reset quaternion is unit only
    to rounding)."""
    m = _model(oracle, substeps=4, episode_len=10 ** 9)
    rng = np.random.default_rng(1)
    b = oracle.Batch(np.arange(6))
    oracle.reset(m, b)
    b.params[14:17] = 0.0          # no current
    b.params[10] = 0.0
    b.params[11:14] = 0.0
    p0 = b.state[0:3].copy()
    q0 = b.state[3:7].copy()
    rew, done, tr = oracle.replay(m, b, np.zeros((300, 8, 6), np.float32), precision, trace=True)
    assert np.all(tr[:, 7:19, :] == 0.0)
    assert np.all(tr[:, 0:3, :] == p0[None])
    q0n = q0 / np.linalg.norm(q0, axis=0)
    tol = 1e-15 if precision == "f64" else 1.2e-7
    assert np.max(np.abs(tr[:, 3:7, :] - q0n[None])) <= tol
    assert not done.any()


def test_quaternion_norm_preserved_fp32(oracle):
    """Unit quaternion to 1e-6 over 10^4 control steps in float arithmetic."""
    m = _model(oracle, substeps=4, episode_len=10 ** 9, dr_enable=1, current_range=0.3)
    b = oracle.Batch(np.arange(4))
    oracle.reset(m, b)
    acts = W.replay_actions(3, 10000, 4, scale=1.0)
    _, _, tr = oracle.replay(m, b, acts, "f32", trace=True)
    qn = np.linalg.norm(tr[:, 3:7, :], axis=1)
    assert np.max(np.abs(qn - 1.0)) <= 1e-6


def test_kinetic_energy_nonincreasing_under_damping(oracle):
    """g = 0, no current, zero thrust: E = 1/2 nu^T M nu never increases."""
    w = W.workload("tiny_64", gravity=(0.0, 0.0, 0.0))
    m = oracle.model(w)
    rng = np.random.default_rng(2)
    M = _mass_diag(w)
    for trial in range(5):
        nu0 = rng.uniform(-1, 1, 6)
        st, pr = oracle.single_env(dict(q=_random_quat(rng), nu=nu0), {})
        e_prev = 0.5 * np.sum(M * st[7:13] ** 2)
        for k in range(400):
            st = oracle.integrate(m, st, pr, np.zeros(6), 0.005, 1)
            e = 0.5 * np.sum(M * st[7:13] ** 2)
            assert e <= e_prev * (1 + 1e-12), (trial, k, e, e_prev)
            e_prev = e
        assert e_prev < 0.5 * np.sum(M * nu0 ** 2)


def test_rotation_of_whole_setup_is_invariant(oracle):
    """Rotate positions, attitudes, goal, gravity and current by one world
    rotation: body velocities and rewards are unchanged, world positions and
    attitudes are rotated."""
    rng = np.random.default_rng(3)
    qw = _random_quat(rng)
    Rw = _rot(qw)
    g = np.array([0.0, 0.0, -9.81])
    mA = _model(oracle, substeps=4, episode_len=10 ** 9)
    mB = oracle.model(W.workload("tiny_64", substeps=4, episode_len=10 ** 9,
                                 gravity=tuple(Rw @ g)))
    n = 5
    bA = oracle.Batch(np.arange(n))
    bA.state[0:3] = rng.uniform(-1, 1, (3, n))
    for i in range(n):
        bA.state[3:7, i] = _random_quat(rng)
        bA.params[3:7, i] = _random_quat(rng)
    bA.state[7:13] = rng.uniform(-0.5, 0.5, (6, n))
    bA.params[0:3] = rng.uniform(-1, 1, (3, n))
    bA.params[7:10] = rng.uniform(0.8, 1.2, (3, n))
    bA.params[10] = rng.uniform(-2, 2, n)
    bA.params[11:14] = rng.uniform(-0.01, 0.01, (3, n))
    bA.params[14:17] = rng.uniform(-0.3, 0.3, (3, n))
    bB = bA.copy()
    bB.state[0:3] = Rw @ bA.state[0:3]
    bB.params[0:3] = Rw @ bA.params[0:3]
    bB.params[14:17] = Rw @ bA.params[14:17]
    for i in range(n):
        bB.state[3:7, i] = _quat_mul(qw, bA.state[3:7, i])
        bB.params[3:7, i] = _quat_mul(qw, bA.params[3:7, i])
    acts = W.replay_actions(4, 60, n)
    rA, _, tA = oracle.replay(mA, bA, acts, trace=True)
    rB, _, tB = oracle.replay(mB, bB, acts, trace=True)
    assert np.allclose(tA[:, 7:19], tB[:, 7:19], rtol=0, atol=1e-9)
    assert np.allclose(rA, rB, rtol=0, atol=1e-9)
    assert np.allclose(np.einsum("ij,tjn->tin", Rw, tA[:, 0:3]), tB[:, 0:3], atol=1e-9)
    for t in (0, 30, 59):
        for i in range(n):
            qa = _quat_mul(qw, tA[t, 3:7, i])
            qb = tB[t, 3:7, i]
            assert min(np.abs(qa - qb).max(), np.abs(qa + qb).max()) < 1e-9


# ----------------------------------------------------------------------------
# Integrator against a brute-force RK4
# ----------------------------------------------------------------------------
def test_semi_implicit_euler_converges_first_order_to_rk4(oracle):
    rng = np.random.default_rng(4)
    m = _model(oracle)
    st, pr = oracle.single_env(
        dict(p=[0.1, -0.2, 0.3], q=_random_quat(rng), nu=rng.uniform(-0.6, 0.6, 6)),
        dict(p_d=[0, 0, 0], s_m=1.1, s_a=0.9, s_d=1.05, dB=1.5, r_b=[0.004, -0.003, 0.008],
             V_c=[0.2, -0.1, 0.05]))
    tau = np.array([20.0, -10.0, 15.0, 0.5, -0.4, 0.8])
    T = 0.2
    ref = oracle.integrate(m, st, pr, tau, 1e-4, 2000, method="rk4")
    ref2 = oracle.integrate(m, st, pr, tau, 5e-5, 4000, method="rk4")
    assert np.max(np.abs(ref[:13] - ref2[:13])) < 1e-10      # RK4 itself converged
    errs = []
    for h in (0.01, 0.005, 0.0025, 0.00125):
        out = oracle.integrate(m, st, pr, tau, h, int(round(T / h)))
        errs.append(np.max(np.abs(out[:13] - ref[:13])))
    ratios = [errs[i] / errs[i + 1] for i in range(3)]
    assert all(1.7 < r < 2.3 for r in ratios), (errs, ratios)
    assert errs[-1] < 2e-3


# ----------------------------------------------------------------------------
# 1-DOF closed forms
# ----------------------------------------------------------------------------
@pytest.mark.parametrize("axis", range(6))
def test_single_axis_decay_matches_bernoulli_solution(oracle, axis):
    """x' = -(a x + b |x| x)/M has x(t) = a x0 e^{-a t/M} / (a + b x0 (1 - e^{-a t/M}))
    for x0 > 0.  Single-axis motion has no Coriolis coupling."""
    w = W.workload("tiny_64")
    m = oracle.model(w)
    Mk = _mass_diag(w)[axis]
    a, b = w["damp_lin"][axis], w["damp_quad"][axis]
    x0 = 0.8
    nu0 = np.zeros(6)
    nu0[axis] = x0
    st, pr = oracle.single_env(dict(nu=nu0), {})
    errs = []
    for h in (2e-4, 1e-4):
        t_end = 1.0
        out = oracle.integrate(m, st, pr, np.zeros(6), h, int(round(t_end / h)))
        e = math.exp(-a * t_end / Mk)
        exact = a * x0 * e / (a + b * x0 * (1 - e))
        others = np.delete(out[7:13], axis)
        assert np.all(others == 0.0)
        errs.append(abs(out[7 + axis] - exact))
    assert errs[1] < 1e-4 * x0
    assert 1.6 < errs[0] / errs[1] < 2.4


def test_terminal_surge_velocity_under_constant_thrust(oracle):
    """The four horizontal thrusters at the same command give pure surge
    force F = 4 * 40 * c / sqrt(2); the speed settles at the root of
    a u + b u^2 = F."""
    w = W.workload("tiny_64", substeps=4, episode_len=10 ** 9)
    m = oracle.model(w)
    c = 0.5
    act = np.zeros((1, 8), np.float32)
    act[0, :4] = c
    tau = oracle.allocate(m, act[0].astype(np.float64))
    F = 4 * 40.0 * c / math.sqrt(2)
    assert np.allclose(tau, [F, 0, 0, 0, 0, 0], atol=1e-12)
    b = oracle.Batch([0])
    b.state[3] = 1.0
    b.params[3] = 1.0
    b.params[7:10] = 1.0
    acts = np.repeat(act[None, :, :].transpose(0, 2, 1), 1500, axis=0)  # [T][8][1]
    oracle.replay(m, b, acts)
    a_l, b_q = w["damp_lin"][0], w["damp_quad"][0]
    u_star = (-a_l + math.sqrt(a_l ** 2 + 4 * b_q * F)) / (2 * b_q)
    assert abs(b.state[7, 0] - u_star) < 1e-6 * u_star
    assert np.all(np.abs(b.state[8:13, 0]) < 1e-12)


def test_heave_acceleration_from_buoyancy_offset(oracle):
    w = W.workload("tiny_64")
    m = oracle.model(w)
    for s_m, s_a, dB in ((1.0, 1.0, 1.5), (1.1, 0.9, -2.0)):
        st, pr = oracle.single_env({}, dict(s_m=s_m, s_a=s_a, dB=dB))
        acc = oracle.nu_dot(m, st, pr, np.zeros(6))
        expect = dB / (s_m * w["mass"] + s_a * w["added_mass"][2])
        assert math.isclose(acc[2], expect, rel_tol=1e-12)
        assert np.all(acc[[0, 1, 3, 4, 5]] == 0.0)


def test_pendulum_period_with_centre_of_buoyancy_above_gravity(oracle):
    """CoB z_b above the CoG restores roll: small oscillations have angular
    frequency sqrt(B z_b / (I_x + A_44)) with B = m g (neutral)."""
    w = W.workload("tiny_64", **NO_DAMP)
    m = oracle.model(w)
    z_b = 0.02
    phi0 = 0.02
    q0 = [math.cos(phi0 / 2), math.sin(phi0 / 2), 0.0, 0.0]
    st, pr = oracle.single_env(dict(q=q0), dict(r_b=[0, 0, z_b]))
    B = w["mass"] * 9.81
    omega = math.sqrt(B * z_b / (w["inertia"][0] + w["added_mass"][3]))
    period = 2 * math.pi / omega
    h = 2e-4
    rolls, ts = [], []
    for k in range(int(2.2 * period / h)):
        st = oracle.integrate(m, st, pr, np.zeros(6), h, 1)
        q = st[3:7]
        rolls.append(math.atan2(2 * (q[0] * q[1] + q[2] * q[3]), 1 - 2 * (q[1] ** 2 + q[2] ** 2)))
        ts.append((k + 1) * h)
    rolls = np.array(rolls)
    # downward zero crossings, linearly interpolated
    idx = np.where((rolls[:-1] > 0) & (rolls[1:] <= 0))[0]
    tc = [ts[i] + h * rolls[i] / (rolls[i] - rolls[i + 1]) for i in idx]
    assert len(tc) >= 2
    measured = tc[1] - tc[0]
    assert abs(measured - period) / period < 2e-3
    assert np.max(np.abs(rolls)) < phi0 * 1.01     # bounded: restoring, not divergent


def test_constant_spin_follows_exponential(oracle):
    """No damping, torque-free spin about a principal axis: the attitude is
    q0 (x) (cos(w t / 2), sin(w t / 2) axis) exactly (the exponential map is
    exact for constant w)."""
    w = W.workload("tiny_64", **NO_DAMP)
    m = oracle.model(w)
    rng = np.random.default_rng(6)
    q0 = _random_quat(rng)
    for axis in range(3):
        nu0 = np.zeros(6)
        nu0[3 + axis] = 1.3
        st, pr = oracle.single_env(dict(q=q0, nu=nu0), {})
        out = oracle.integrate(m, st, pr, np.zeros(6), 0.005, 400)
        t = 2.0
        dq = np.zeros(4)
        dq[0] = math.cos(1.3 * t / 2)
        dq[1 + axis] = math.sin(1.3 * t / 2)
        assert np.allclose(out[3:7], _quat_mul(q0, dq), atol=1e-12)
        assert np.allclose(out[7:13], nu0, atol=0)


# ----------------------------------------------------------------------------
# Coriolis structure: Kirchhoff's equations and the Munk moment
# ----------------------------------------------------------------------------
def _impulses(w, st):
    M = _mass_diag(w)
    R = _rot(st[3:7])
    P = R @ (M[:3] * st[7:10])
    L = R @ (M[3:] * st[10:13]) + np.cross(st[0:3], P)
    E = 0.5 * np.sum(M * st[7:13] ** 2)
    return P, L, E


def test_kirchhoff_impulses_conserved_in_ideal_fluid(oracle):
    """No damping, no gravity, no current, no thrust: a body in ideal fluid
    conserves its world-frame linear impulse R (m + A1) v, its angular impulse
    R (I + A2) w + p x R (m + A1) v, and its energy (Kirchhoff / Lamb).  Drift
    is first order in h and vanishes as h -> 0."""
    w = W.workload("tiny_64", gravity=(0.0, 0.0, 0.0), inertia=(0.10, 0.20, 0.30), **NO_DAMP)
    m = oracle.model(w)
    rng = np.random.default_rng(7)
    st, pr = oracle.single_env(dict(p=[0.3, -0.2, 0.1], q=_random_quat(rng),
                                    nu=[0.6, -0.4, 0.3, 0.8, -0.5, 0.6]), {})
    P0, L0, E0 = _impulses(w, st)
    drifts = []
    for h in (4e-4, 2e-4):
        out = oracle.integrate(m, st, pr, np.zeros(6), h, int(round(1.0 / h)))
        P, L, E = _impulses(w, out)
        drifts.append(max(np.abs(P - P0).max() / np.abs(P0).max(),
                          np.abs(L - L0).max() / np.abs(L0).max(), abs(E - E0) / E0))
    assert drifts[1] < 2e-3
    assert 1.6 < drifts[0] / drifts[1] < 2.4, drifts
    # the motion is genuinely coupled: body velocities change a lot
    assert np.abs(out[7:13] - st[7:13]).max() > 0.1


def test_munk_moment_turns_body_broadside(oracle):
    """A body translating obliquely (u, v > 0) with sway added mass above surge
    added mass feels the yaw moment (A11 - A22) u v, which turns it away from
    its direction of motion (Munk)."""
    w = W.workload("tiny_64", **NO_DAMP)
    m = oracle.model(w)
    u, v = 0.5, 0.3
    st, pr = oracle.single_env(dict(nu=[u, v, 0, 0, 0, 0]), {})
    acc = oracle.nu_dot(m, st, pr, np.zeros(6))
    A11, A22 = w["added_mass"][0], w["added_mass"][1]
    Iz = w["inertia"][2] + w["added_mass"][5]
    assert acc[5] < 0
    assert math.isclose(acc[5] * Iz, (A11 - A22) * u * v, rel_tol=1e-12)
    assert acc[0] == 0 and acc[1] == 0


def test_free_rigid_body_translates_in_a_straight_line(oracle):
    """No fluid (no added mass, no damping), no gravity: a spinning body keeps
    its world-frame velocity (the m w x v term cancels the frame rotation)."""
    w = W.workload("tiny_64", gravity=(0.0, 0.0, 0.0), added_mass=(0.0,) * 6, **NO_DAMP)
    m = oracle.model(w)
    st, pr = oracle.single_env(dict(nu=[0.5, 0.0, 0.0, 0.0, 0.0, 1.0]), {})
    errs = []
    for h in (1e-3, 5e-4):
        out = oracle.integrate(m, st, pr, np.zeros(6), h, int(round(1.0 / h)))
        Vw = _rot(out[3:7]) @ out[7:10]
        errs.append(max(np.abs(Vw - [0.5, 0, 0]).max(), np.abs(out[0:3] - [0.5, 0, 0]).max()))
    assert errs[1] < 1e-3
    assert 1.6 < errs[0] / errs[1] < 2.4


# ----------------------------------------------------------------------------
# Current: Galilean invariance
# ----------------------------------------------------------------------------
def test_uniform_current_is_a_galilean_shift(oracle):
    """With a uniform current V_c the motion relative to the water is the
    no-current motion: p_c(t) = p_0(t) + V_c t, same attitude, and
    nu_c - [R^T V_c; 0] = nu_0 (up to the integrator's O(h) error)."""
    rng = np.random.default_rng(8)
    m = _model(oracle)
    q0 = _random_quat(rng)
    Vc = np.array([0.25, -0.2, 0.15])
    nu_r0 = np.array([0.3, -0.2, 0.1, 0.4, -0.3, 0.5])
    params = dict(s_m=1.05, s_a=0.95, s_d=1.1, dB=1.0, r_b=[0.003, 0.002, 0.008])
    stA, prA = oracle.single_env(dict(q=q0, nu=nu_r0 + np.r_[_rot(q0).T @ Vc, 0, 0, 0]),
                                 dict(V_c=Vc, **params))
    stB, prB = oracle.single_env(dict(q=q0, nu=nu_r0), params)
    tau = np.array([10.0, 5.0, -8.0, 0.2, 0.3, -0.4])
    errs = []
    for h in (1e-3, 5e-4):
        n = int(round(1.0 / h))
        a = oracle.integrate(m, stA, prA, tau, h, n)
        b = oracle.integrate(m, stB, prB, tau, h, n)
        e_p = np.abs(a[0:3] - (b[0:3] + Vc * 1.0)).max()
        e_q = min(np.abs(a[3:7] - b[3:7]).max(), np.abs(a[3:7] + b[3:7]).max())
        e_nu = np.abs(a[7:13] - np.r_[_rot(a[3:7]).T @ Vc, 0, 0, 0] - b[7:13]).max()
        errs.append(max(e_p, e_q, e_nu))
    assert errs[1] < 2e-3
    assert 1.6 < errs[0] / errs[1] < 2.4, errs
