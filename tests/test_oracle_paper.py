"""Pins for the oracle's paper-model environment (§IV-B of the paper: wrench
action of Eq. 1, inertia-box fluid model, effective gravity, 12-float
axis-angle observation, five-term reward of Eqs. 2-7) against facts fixed
outside its code: the uniform-box inertia formula, closed-form terminal
velocities and rates under drag, exponential viscous decay, gravity rotated
by scipy, torque-free rigid-body invariants, scipy's rotation vectors,
hand-computed reward terms, a numpy moving average, scipy's normal log-density
and first-order convergence of the integrator to an RK4 brute force."""
import math

import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W


def _model(oracle, **over):
    return oracle.paper_model(W.workload("paper_tiny", **over))


def _rot(q):
    from scipy.spatial.transform import Rotation
    return Rotation.from_quat([q[1], q[2], q[3], q[0]])


def _quat_from_rotvec(v):
    from scipy.spatial.transform import Rotation
    x, y, z, w = Rotation.from_rotvec(v).as_quat()
    return np.array([w, x, y, z])


def _random_quat(rng):
    q = rng.standard_normal(4)
    return q / np.linalg.norm(q)


def _box_inertia(mass, sides):
    a, b, c = sides
    return (mass * (b * b + c * c) / 12, mass * (a * a + c * c) / 12, mass * (a * a + b * b) / 12)


SIDES = (0.6, 0.35, 0.25)
MASS = 11.5


def _box_model(oracle, **over):
    return _model(oracle, mass=MASS, inertia=_box_inertia(MASS, SIDES), **over)


def test_box_sides_invert_the_uniform_box_inertia(oracle):
    m = _box_model(oracle)
    assert np.allclose(oracle.paper_box(m), SIDES, rtol=1e-12)


def test_wrench_scaling_and_clip_eq1(oracle):
    m = _model(oracle, f_max=40.0, tau_max=10.0)
    a = np.array([1.5, -0.3, 0.2, -2.0, 0.5, 0.9])
    a_c, tau = oracle.paper_wrench(m, a)
    assert np.array_equal(a_c, [1.0, -0.3, 0.2, -1.0, 0.5, 0.9])
    assert np.allclose(tau, [40.0, -12.0, 8.0, -10.0, 5.0, 9.0], rtol=1e-15)


def test_terminal_surge_velocity_under_drag(oracle):
    """F = 1/2 rho A v^2 + 3 pi mu d v at steady state, A = b_y b_z,
    d = mean side."""
    rho, mu, F = 1000.0, 0.5, 30.0
    m = _box_model(oracle, fluid_density=rho, fluid_viscosity=mu, g_eff=0.0)
    A = SIDES[1] * SIDES[2]
    c = 3 * math.pi * mu * sum(SIDES) / 3
    v_star = (-c + math.sqrt(c * c + 2 * rho * A * F)) / (rho * A)
    st, pr = oracle.paper_single_env({}, {})
    st = oracle.paper_integrate(m, st, pr, [F, 0, 0, 0, 0, 0], 1e-3, 20000)
    assert st[7] == pytest.approx(v_star, rel=1e-6)
    assert np.allclose(st[8:13], 0.0, atol=1e-12)


def test_viscous_decay_is_exponential(oracle):
    """rho = 0: m v' = F - c v with c = 3 pi mu d, v(0) = 0 ->
    v(t) = F/c (1 - exp(-c t / m)); RK4 matches to 1e-9."""
    mu, F, t_end = 2.0, 5.0, 0.8
    m = _box_model(oracle, fluid_density=0.0, fluid_viscosity=mu, g_eff=0.0)
    c = 3 * math.pi * mu * sum(SIDES) / 3
    st, pr = oracle.paper_single_env({}, {})
    st = oracle.paper_integrate(m, st, pr, [0, F, 0, 0, 0, 0], 1e-3, int(t_end / 1e-3),
                                method="rk4")
    assert st[8] == pytest.approx(F / c * (1 - math.exp(-c * t_end / MASS)), rel=1e-9)


def test_terminal_roll_rate_under_drag(oracle):
    """tau = rho/64 b_x (b_y^4 + b_z^4) w^2 + pi mu d^3 w at steady state."""
    rho, mu, tau = 1000.0, 0.5, 0.4
    m = _box_model(oracle, fluid_density=rho, fluid_viscosity=mu, g_eff=0.0)
    bx, by, bz = SIDES
    k2 = rho / 64 * bx * (by ** 4 + bz ** 4)
    k1 = math.pi * mu * (sum(SIDES) / 3) ** 3
    w_star = (-k1 + math.sqrt(k1 * k1 + 4 * k2 * tau)) / (2 * k2)
    st, pr = oracle.paper_single_env({}, {})
    st = oracle.paper_integrate(m, st, pr, [0, 0, 0, tau, 0, 0], 1e-3, 40000)
    assert st[10] == pytest.approx(w_star, rel=1e-6)


def test_effective_gravity_in_the_body_frame(oracle):
    rng = np.random.default_rng(3)
    m = _model(oracle)
    for g in (0.3, -0.15):
        q = _random_quat(rng)
        st, pr = oracle.paper_single_env({"q": q}, {"g_eff": g})
        acc = oracle.paper_nu_dot(m, st, pr, np.zeros(6))
        expect = _rot(q).apply([0.0, 0.0, -g], inverse=True)
        assert np.allclose(acc[:3], expect, atol=1e-14)
        assert np.allclose(acc[3:], 0.0, atol=1e-15)


def test_torque_free_rigid_body_invariants(oracle):
    """No fluid, no gravity: world angular momentum R I w and kinetic energy
    are conserved (RK4), and the body moves in a straight line."""
    m = _box_model(oracle, fluid_density=0.0, fluid_viscosity=0.0, g_eff=0.0)
    I = np.array(_box_inertia(MASS, SIDES))
    w0 = np.array([0.7, 2.0, -0.4])
    v0 = np.array([0.3, -0.2, 0.1])
    st, pr = oracle.paper_single_env({"nu": np.r_[v0, w0]}, {})
    L0 = I * w0
    E0 = 0.5 * np.dot(I * w0, w0)
    p_world0 = v0.copy()
    st = oracle.paper_integrate(m, st, pr, np.zeros(6), 1e-3, 3000, method="rk4")
    q, w = st[3:7], st[10:13]
    R = _rot(q)
    assert np.allclose(R.apply(I * w), L0, atol=1e-9)
    assert 0.5 * np.dot(I * w, w) == pytest.approx(E0, rel=1e-9)
    # linear momentum: world velocity stays v0 (straight line from the origin)
    assert np.allclose(st[0:3], p_world0 * 3.0, atol=1e-8)


def test_integrator_converges_first_order_to_rk4(oracle):
    m = _box_model(oracle, fluid_density=1000.0, fluid_viscosity=0.01, g_eff=0.4)
    rng = np.random.default_rng(5)
    st0, pr = oracle.paper_single_env({"q": _random_quat(rng),
                                       "nu": rng.uniform(-0.5, 0.5, 6)}, {"g_eff": 0.4})
    tau = [10.0, -5.0, 3.0, 0.5, -0.3, 0.2]
    ref = oracle.paper_integrate(m, st0, pr, tau, 1e-4, 5000, method="rk4")
    errs = []
    for h in (4e-3, 2e-3, 1e-3):
        s = oracle.paper_integrate(m, st0, pr, tau, h, int(round(0.5 / h)))
        errs.append(np.max(np.abs(s[:13] - ref[:13])))
    assert 1.7 < errs[0] / errs[1] < 2.3 and 1.7 < errs[1] / errs[2] < 2.3


def test_observation_matches_scipy(oracle):
    from scipy.spatial.transform import Rotation
    rng = np.random.default_rng(11)
    for _ in range(50):
        q, qd = _random_quat(rng), _random_quat(rng)
        p, pd, nu = rng.uniform(-2, 2, 3), rng.uniform(-2, 2, 3), rng.uniform(-1, 1, 6)
        st, pr = oracle.paper_single_env({"p": p, "q": q, "nu": nu}, {"p_d": pd, "q_d": qd})
        obs = oracle.paper_observe(st, pr)
        assert np.allclose(obs[0:3], _rot(q).apply(p - pd, inverse=True), atol=1e-12)
        rv = (_rot(qd).inv() * _rot(q)).as_rotvec()
        assert np.allclose(obs[3:6], rv, atol=1e-10)
        assert np.array_equal(obs[6:12], nu)


def test_observation_special_attitudes(oracle):
    rng = np.random.default_rng(12)
    q = _random_quat(rng)
    # the same rotation with either quaternion sign, and the identity
    for qd in (q, -q):
        st, pr = oracle.paper_single_env({"q": q}, {"q_d": qd})
        assert np.allclose(oracle.paper_observe(st, pr)[3:6], 0.0, atol=1e-12)
    # a half turn about a known axis: the vector has length pi along the axis
    axis = np.array([1.0, 2.0, -2.0]) / 3.0
    qh = np.r_[0.0, axis]
    st, pr = oracle.paper_single_env({"q": qh}, {})
    th = oracle.paper_observe(st, pr)[3:6]
    assert np.linalg.norm(th) == pytest.approx(math.pi, rel=1e-12)
    assert abs(np.dot(th / math.pi, axis)) == pytest.approx(1.0, rel=1e-12)
    # a small rotation: the vector is the rotation vector, not zero
    small = _quat_from_rotvec([1e-9, -2e-9, 3e-9])
    st, pr = oracle.paper_single_env({"q": small}, {})
    assert np.allclose(oracle.paper_observe(st, pr)[3:6], [1e-9, -2e-9, 3e-9], rtol=1e-9)


def test_reward_terms_by_hand(oracle):
    """Eqs. (2)-(7) with every weight distinct; identity attitude so the
    body-frame position error is p - p_d."""
    wts = dict(w_pos=0.7, w_axes=(1.0, 2.0, 3.0), w_att=0.5, w_act=0.03, w_vel=0.2,
               w_mavg=0.4, mavg_len=3)
    m = _model(oracle, **wts)
    p, pd = np.array([1.0, 0.5, -2.0]), np.zeros(3)
    ang = 0.4
    qd = np.array([math.cos(ang / 2), 0.0, 0.0, math.sin(ang / 2)])
    nu = np.array([0.1, -0.2, 0.3, 0.5, -0.25, 0.75])
    hist = np.zeros((8, 6))
    hist[0] = [0.3, 0.0, -0.6, 0.9, 0.0, 0.3]
    hist[1] = [0.0, 0.3, 0.0, -0.3, 0.6, 0.0]
    hist[2] = [0.6, 0.3, 0.3, 0.0, 0.0, 0.3]
    hist[3] = 100.0                       # beyond K = 3: must not count
    st, pr = oracle.paper_single_env({"p": p, "nu": nu, "hist": hist}, {"p_d": pd, "q_d": qd})
    a_c = np.array([0.5, -0.5, 0.25, 0.1, -0.2, 0.3])
    r = oracle.paper_reward(m, st, pr, a_c)
    r_pos = -0.7 * ((1 * 1.0) ** 2 + (2 * 0.5) ** 2 + (3 * -2.0) ** 2)
    r_att = -0.5 * ang ** 2
    r_act = -0.03 * (0.1 ** 2 + 0.2 ** 2 + 0.3 ** 2)
    r_vel = -0.2 * (0.5 ** 2 + 0.25 ** 2 + 0.75 ** 2)
    mean = hist[:3].mean(axis=0)
    r_mavg = -0.4 * np.sum((a_c - mean) ** 2)
    assert r == pytest.approx(r_pos + r_att + r_act + r_vel + r_mavg, rel=1e-13)


def test_moving_average_over_a_replay(oracle):
    """Only the r_act-mavg term on: the reward is -||a_c,t - mean of the K
    previous clipped actions||^2 (zeros before step K and after a reset)."""
    K, L, n, T = 3, 7, 5, 16
    w = W.workload("paper_tiny", w_pos=0.0, w_att=0.0, w_act=0.0, w_vel=0.0, w_mavg=1.0,
                   mavg_len=K, episode_len=L)
    m = oracle.paper_model(w)
    b = oracle.PaperBatch(np.arange(n))
    oracle.paper_reset(m, b)
    acts = W.replay_actions(2, T, n, scale=1.2, act=6)
    rew, done, _ = oracle.paper_replay(m, b, acts)
    a_c = np.clip(acts.astype(np.float64), -1, 1)
    for i in range(n):
        hist = []
        for t in range(T):
            prev = hist[-K:]
            mean = np.sum(prev, axis=0) / K if prev else np.zeros(6)
            assert rew[t, i] == pytest.approx(-np.sum((a_c[t, :, i] - mean) ** 2), rel=1e-12,
                                              abs=1e-15)
            hist.append(a_c[t, :, i])
            if (t + 1) % L == 0:
                assert done[t, i] == 1
                hist = []
            else:
                assert done[t, i] == 0


def test_reset_draws(oracle):
    from scipy.spatial.transform import Rotation
    n = 400
    w = W.workload("paper_tiny", dr_enable=1, g_eff=0.1, dr_gravity_range=0.2,
                   init_pos_range=0.5, init_att_range=0.2)
    m = oracle.paper_model(w)
    b = oracle.PaperBatch(np.arange(n))
    oracle.paper_reset(m, b)
    assert np.all(np.abs(b.params[0:3]) <= 2.0) and np.all(np.abs(b.state[0:3]) <= 0.5)
    assert np.all(np.abs(b.params[7] - 0.1) <= 0.2 + 1e-7)
    assert np.ptp(b.params[7]) > 0.3                     # the offset is actually drawn
    assert np.all(b.state[7:] == 0.0) and np.all(b.episode == 1) and np.all(b.t_ep == 0)
    # goal attitude: Z-Y-X Euler angles from uniforms 3..5 of the reset stream
    r = math.pi / 3
    for i in range(0, n, 37):
        words = np.concatenate([oracle.philox(i, 0, [0, 0, 1, blk]) for blk in range(2)])
        u = [oracle.lib().oracle_word_to_uniform(int(x)) for x in words[:8]]
        roll, pitch, yaw = (ui * 2 * r - r for ui in u[3:6])
        x, y, z, wq = Rotation.from_euler("ZYX", [yaw, pitch, roll]).as_quat()
        qd = b.params[3:7, i]
        assert np.allclose(qd, [wq, x, y, z], atol=2e-7) or np.allclose(qd, [-wq, -x, -y, -z],
                                                                       atol=2e-7)
    # DR off: the nominal effective gravity
    m0 = oracle.paper_model(W.workload("paper_tiny", g_eff=0.1))
    b0 = oracle.PaperBatch(np.arange(8))
    oracle.paper_reset(m0, b0)
    assert np.all(b0.params[7] == np.float32(0.1))


def test_rollout_log_probability_and_dones(oracle):
    from scipy.stats import norm
    n, T, L = 6, 9, 4
    w = W.workload("paper_tiny", episode_len=L, logstd_fixed=(-0.5, 0.0, 0.3, -1.0, 0.1, 0.2))
    m = oracle.paper_model(w)
    b = oracle.PaperBatch(np.arange(n))
    oracle.paper_reset(m, b)
    pw = W.policy_weights(w)
    out = oracle.paper_rollout(m, b, pw, None, 100, T)
    ls = np.array(w["logstd_fixed"], dtype=np.float32).astype(np.float64)   # stored as float
    for t in range(T):
        mu = oracle.mlp(pw, 12, w["hidden"], 6, False, out["obs"][t].T)
        for i in range(n):
            eps = oracle.normals(i, 0, 100 + t)[:6]
            a = mu[i] + np.exp(ls) * eps
            assert np.allclose(out["act"][t, :, i], a, rtol=1e-12, atol=1e-14)
            lp = np.sum(norm.logpdf(a, loc=mu[i], scale=np.exp(ls)))
            assert out["logp"][t, i] == pytest.approx(lp, rel=1e-12)
    assert np.array_equal(out["done"][:, 0], [(t + 1) % L == 0 for t in range(T)])


def _golden_setup():
    import os
    vals = {}
    with open(os.path.join(os.path.dirname(__file__), "golden", "paper_setup.txt")) as f:
        for line in f:
            line = line.split("#", 1)[0].split()
            if line:
                vals[line[0]] = float(line[1])
    return vals


def test_golden_paper_setup(oracle):
    """The task constants the paper prints (golden/paper_setup.txt, each line
    cited: §IV-A, §IV-B1, §IV-B2, §V-A1) against the 4,096-env paper workload
    and the oracle's reset draws for it: observation and action widths, the
    action bound, env count, episode length, and references within [-2, 2] m
    and [-60, 60] degrees per axis, each range used in full."""
    from scipy.spatial.transform import Rotation
    g = _golden_setup()
    w = W.workload("paper_4096")
    assert W.obs_dim(w) == g["obs_dim"] and W.act_dim(w) == g["act_dim"]
    assert w["n_envs"] == g["n_envs"] and w["episode_len"] == g["episode_len"]
    m = oracle.paper_model(w)
    bound = g["action_bound"]
    a_c, tau = oracle.paper_wrench(m, np.array([3.0, -3.0, 0.5, 3.0, -3.0, -0.5]))
    assert np.array_equal(a_c, [bound, -bound, 0.5, bound, -bound, -0.5])
    assert np.allclose(tau[[0, 3]], [w["f_max"], w["tau_max"]], rtol=1e-15)
    b = oracle.PaperBatch(np.arange(int(g["n_envs"])))
    oracle.paper_reset(m, b)
    pd = b.params[0:3]
    assert np.all(np.abs(pd) <= g["goal_pos_range_m"])
    assert np.all(np.abs(pd).max(axis=1) > 0.99 * g["goal_pos_range_m"])
    qd = b.params[3:7]
    yaw_pitch_roll = Rotation.from_quat(np.stack([qd[1], qd[2], qd[3], qd[0]], axis=1)).as_euler(
        "ZYX", degrees=True)
    assert np.all(np.abs(yaw_pitch_roll) <= g["goal_att_range_deg"] + 1e-4)
    assert np.all(np.abs(yaw_pitch_roll).max(axis=0) > 0.99 * g["goal_att_range_deg"])
