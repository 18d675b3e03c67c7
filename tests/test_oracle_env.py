"""Pins for the oracle's environment logic: observation and reward on
hand-computed cases, thruster allocation against the thruster geometry,
reset draws against scipy's Euler-angle conversion and the draw ranges, the
networks against numpy / torch CPU, and the rollout's bookkeeping (done
flags, auto-reset, log-probabilities against scipy's normal log-density)."""
import math

import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W


def _yaw_quat(psi):
    return [math.cos(psi / 2), 0.0, 0.0, math.sin(psi / 2)]


# ----------------------------------------------------------------------------
# Observation and reward
# ----------------------------------------------------------------------------
def test_observation_for_a_yawed_vehicle(oracle):
    """Vehicle yawed +90 deg at (1, 0, 0), goal at the origin with zero yaw.
    The goal-to-vehicle offset (1, 0, 0) lies on the vehicle's right: body
    (0, -1, 0).  R_e = R(q_d)^T R(q) = R_z(90), whose columns are the body
    axes in the goal frame: x -> (0, 1, 0), y -> (-1, 0, 0), z -> (0, 0, 1);
    the geodesic error is pi/2."""
    st, pr = oracle.single_env(dict(p=[1, 0, 0], q=_yaw_quat(math.pi / 2),
                                    nu=[0.1, 0.2, 0.3, 0.4, 0.5, 0.6]), dict(p_d=[0, 0, 0]))
    obs, theta = oracle.observe(st, pr)
    assert np.allclose(obs[0:3], [0, -1, 0], atol=1e-15)
    Re_cols = obs[3:12].reshape(3, 3)          # rows = columns of R_e
    assert np.allclose(Re_cols[0], [0, 1, 0], atol=1e-15)
    assert np.allclose(Re_cols[1], [-1, 0, 0], atol=1e-15)
    assert np.allclose(Re_cols[2], [0, 0, 1], atol=1e-15)
    assert np.allclose(obs[12:18], [0.1, 0.2, 0.3, 0.4, 0.5, 0.6])
    assert math.isclose(theta, math.pi / 2, rel_tol=1e-14)


def test_attitude_error_matches_rotation_matrix_definitions(oracle):
    """Random attitudes: R_e from the observation equals R(q_d)^T R(q) built by
    scipy; the geodesic angle equals arccos((tr R_e - 1) / 2) and scipy's
    relative-rotation magnitude; the position error is R(q)^T (p - p_d)."""
    from scipy.spatial.transform import Rotation
    rng = np.random.default_rng(0)
    for _ in range(50):
        q = rng.standard_normal(4)
        q /= np.linalg.norm(q)
        qd = rng.standard_normal(4)
        qd /= np.linalg.norm(qd)
        p, pd = rng.uniform(-2, 2, 3), rng.uniform(-2, 2, 3)
        st, pr = oracle.single_env(dict(p=p, q=q), dict(p_d=pd, q_d=qd))
        obs, theta = oracle.observe(st, pr)
        Rq = Rotation.from_quat([q[1], q[2], q[3], q[0]])
        Rd = Rotation.from_quat([qd[1], qd[2], qd[3], qd[0]])
        Re = Rd.as_matrix().T @ Rq.as_matrix()
        assert np.allclose(obs[3:12], Re.T.reshape(-1), atol=1e-13)   # column-major
        assert np.allclose(obs[0:3], Rq.as_matrix().T @ (p - pd), atol=1e-13)
        ang = (Rd.inv() * Rq).magnitude()
        assert math.isclose(theta, ang, abs_tol=1e-9)
        c = np.clip((np.trace(Re) - 1) / 2, -1, 1)
        if 0.05 < theta < math.pi - 0.05:
            assert math.isclose(theta, math.acos(c), abs_tol=1e-9)


def test_reward_terms(oracle):
    """r = -w_pos ||dp|| - w_att theta_e - w_act ||a_c||^2 - w_vs ||nu - nu_prev||^2."""
    w = W.workload("tiny_64", w_vs=0.25)
    m = oracle.model(w)
    st, pr = oracle.single_env(dict(p=[3, 4, 0], q=_yaw_quat(math.pi / 3),
                                    nu=[1, 0, 0, 0, 0, 0], nu_prev=[0, 0, 0, 0, 0, 2]),
                               dict(p_d=[0, 0, 0]))
    a_c = np.array([1, -1, 0.5, 0, 0, 0, 0, 0.5])
    r = oracle.reward(m, st, pr, a_c)
    expect = -1.0 * 5.0 - 0.5 * (math.pi / 3) - 0.01 * 2.5 - 0.25 * 5.0
    assert math.isclose(r, expect, rel_tol=1e-14)


# ----------------------------------------------------------------------------
# Thruster allocation
# ----------------------------------------------------------------------------
def test_allocation_produces_wrenches_of_the_thruster_layout(oracle):
    m = oracle.model(W.workload("tiny_64"))
    s = 1 / math.sqrt(2)
    F = 40.0
    # all horizontal thrusters forward: pure surge 4 s F
    tau = oracle.allocate(m, np.r_[1, 1, 1, 1, 0, 0, 0, 0])
    assert np.allclose(tau, [4 * s * F, 0, 0, 0, 0, 0], atol=1e-12)
    # all vertical thrusters up: pure heave 4 F
    tau = oracle.allocate(m, np.r_[0, 0, 0, 0, 1, 1, 1, 1])
    assert np.allclose(tau, [0, 0, 4 * F, 0, 0, 0], atol=1e-12)
    # left verticals up, right verticals down: pure roll moment 4 * 0.22 F
    tau = oracle.allocate(m, np.r_[0, 0, 0, 0, 1, -1, 1, -1])
    assert np.allclose(tau, [0, 0, 0, 4 * 0.22 * F, 0, 0], atol=1e-12)
    # front verticals up, rear down: nose-up pitch is a negative moment about +y
    tau = oracle.allocate(m, np.r_[0, 0, 0, 0, 1, 1, -1, -1])
    assert np.allclose(tau, [0, 0, 0, 0, -4 * 0.12 * F, 0], atol=1e-12)
    # the yaw pair pattern: pure yaw moment 4 * 0.25 s F
    tau = oracle.allocate(m, np.r_[-1, 1, -1, 1, 0, 0, 0, 0])
    assert np.allclose(tau, [0, 0, 0, 0, 0, 4 * 0.25 * s * F], atol=1e-12)
    # clipping at +-1
    assert np.allclose(oracle.allocate(m, np.r_[5, 5, 5, 5, 0, 0, 0, 0]),
                       oracle.allocate(m, np.r_[1, 1, 1, 1, 0, 0, 0, 0]))
    assert np.linalg.matrix_rank(W.allocation_matrix()) == 6


# ----------------------------------------------------------------------------
# Reset draws
# ----------------------------------------------------------------------------
def test_reset_draws_follow_ranges_and_euler_convention(oracle):
    from scipy.spatial.transform import Rotation
    w = W.workload("dr_16384")
    m = oracle.model(w)
    n = 2000
    b = oracle.Batch(np.arange(n))
    oracle.reset(m, b)
    st, pr = b.state, b.params
    assert np.all(np.abs(st[0:3]) <= 0.5) and np.all(np.abs(pr[0:3]) <= 1.0)
    assert np.all(st[7:19] == 0) and np.all(b.t_ep == 0) and np.all(b.episode == 1)
    assert np.all((pr[7:10] >= 0.8) & (pr[7:10] <= 1.2))
    assert np.all(np.abs(pr[10]) <= 2.0) and np.all(np.abs(pr[11:14]) <= 0.01)
    assert np.all(np.abs(pr[14:17]) <= np.float32(0.3))
    # attitude: |roll|, |pitch|, |yaw| <= 0.3 under the intrinsic Z-Y-X convention
    qs = st[3:7].T
    assert np.allclose(np.linalg.norm(qs, axis=1), 1, atol=3e-7)
    eul = Rotation.from_quat(qs[:, [1, 2, 3, 0]]).as_euler("ZYX")
    assert np.all(np.abs(eul) <= 0.3 + 1e-6)
    # goal attitude: yaw only, spanning (-pi, pi)
    assert np.all(pr[4:6] == 0)
    gyaw = 2 * np.arctan2(pr[6], pr[3])
    assert gyaw.min() < -2.8 and gyaw.max() > 2.8
    # uniformity of the goal position draw (KS)
    stats = pytest.importorskip("scipy.stats")
    assert stats.kstest(pr[0], stats.uniform(-1, 2).cdf).pvalue > 1e-3


def test_reset_euler_angles_match_drawn_uniforms(oracle):
    """The attitude of a reset is the Z-Y-X composition of the drawn roll,
    pitch and yaw (uniforms 3, 4, 5 of the reset stream), checked against
    scipy's Euler conversion."""
    from scipy.spatial.transform import Rotation
    L = oracle.lib()
    w = W.workload("tiny_64")
    m = oracle.model(w)
    for env in (0, 5, 123456):
        b = oracle.Batch([env])
        b.episode[:] = 7
        oracle.reset(m, b)
        words = np.concatenate([oracle.philox(env, 0, [7, 0, 1, k]) for k in range(5)])
        u = [L.oracle_word_to_uniform(int(x)) for x in words]
        r = np.float32(0.3)
        ang = [np.float32(u[3 + k]) * (r + r) - r for k in range(3)]   # roll, pitch, yaw
        q = b.state[3:7, 0]
        eul = Rotation.from_quat([q[1], q[2], q[3], q[0]]).as_euler("ZYX")
        assert np.allclose(eul[::-1], ang, atol=1e-6)
        assert np.allclose(b.state[0:3, 0],
                           [np.float32(u[k]) * np.float32(1.0) - np.float32(0.5) for k in range(3)],
                           atol=1e-7)
        assert b.episode[0] == 8


def test_reset_is_deterministic_per_env_and_episode(oracle):
    m = oracle.model(W.workload("dr_16384"))
    b1 = oracle.Batch([3, 4])
    b2 = oracle.Batch([3, 4])
    oracle.reset(m, b1)
    oracle.reset(m, b2)
    assert np.array_equal(b1.state, b2.state) and np.array_equal(b1.params, b2.params)
    oracle.reset(m, b2)           # next episode
    assert not np.array_equal(b1.state[0:3], b2.state[0:3])
    assert not np.array_equal(b1.state[:, 0], b1.state[:, 1])


# ----------------------------------------------------------------------------
# Networks
# ----------------------------------------------------------------------------
def _np_mlp(wts, in_dim, hidden, out_dim, x):
    shapes = W.mlp_shapes(in_dim, hidden, out_dim)
    parts, off = {}, 0
    for name, shp in shapes:
        k = int(np.prod(shp))
        parts[name] = wts[off:off + k].reshape(shp).astype(np.float64)
        off += k
    h1 = np.tanh(x @ parts["W1"].T + parts["b1"])
    h2 = np.tanh(h1 @ parts["W2"].T + parts["b2"])
    return h2 @ parts["W3"].T + parts["b3"]


@pytest.mark.parametrize("hidden,out_dim", [(64, 8), (256, 16), (256, 1)])
def test_mlp_fp32_matches_numpy(oracle, hidden, out_dim):
    wts = W.mlp_weights(0, 18, hidden, out_dim, bias_std=0.1)
    x = W.random_observations(1, 64).astype(np.float64)
    got = oracle.mlp(wts, 18, hidden, out_dim, False, x)
    ref = _np_mlp(wts, 18, hidden, out_dim, x)
    assert np.allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_mlp_bf16_matches_torch_emulation(oracle):
    """bf16 mode = bf16 weights and inputs, exact accumulation, fp32 bias, tanh,
    activations rounded to bf16; emulated with torch CPU bf16 casts."""
    torch = pytest.importorskip("torch")
    hidden, out_dim = 256, 16
    wts = W.mlp_weights(0, 18, hidden, out_dim, bias_std=0.1)
    x = W.random_observations(2, 64).astype(np.float64)
    shapes = W.mlp_shapes(18, hidden, out_dim)
    P, off = {}, 0
    for name, shp in shapes:
        k = int(np.prod(shp))
        t = torch.from_numpy(wts[off:off + k].reshape(shp).copy())
        P[name] = (t.to(torch.bfloat16).to(torch.float64) if name.startswith("W")
                   else t.to(torch.float64))
        off += k
    bf = lambda t: t.to(torch.bfloat16).to(torch.float64)
    xt = bf(torch.from_numpy(x))
    h1 = bf(torch.tanh(xt @ P["W1"].T + P["b1"]))
    h2 = bf(torch.tanh(h1 @ P["W2"].T + P["b2"]))
    ref = (h2 @ P["W3"].T + P["b3"]).numpy()
    got = oracle.mlp(wts, 18, hidden, out_dim, True, x)
    # the torch emulation rounds tanh(float64) to bf16 the same way; any
    # difference comes from an activation within 1e-12 of a bf16 tie
    assert np.allclose(got, ref, rtol=0, atol=1e-9)


# ----------------------------------------------------------------------------
# Rollout bookkeeping
# ----------------------------------------------------------------------------
def test_rollout_done_and_auto_reset(oracle):
    """Episodes end exactly every episode_len steps; the step after a done
    starts from the next episode's reset draw."""
    w = W.workload("tiny_64", episode_len=7)
    m = oracle.model(w)
    n = 3
    b = oracle.Batch(np.arange(n))
    oracle.reset(m, b)
    pw = W.policy_weights(w)
    out = oracle.rollout(m, b, pw, None, 0, 20)
    done = out["done"]
    assert np.array_equal(np.where(done[:, 0])[0], [6, 13])
    assert np.all(done == done[:, :1])
    # obs at t = 7 is the observation of the reset state of episode index 1
    fresh = oracle.Batch(np.arange(n))
    fresh.episode[:] = 1
    oracle.reset(m, fresh)
    obs_fresh = np.array([oracle.observe(fresh.state[:, i], fresh.params[:, i])[0]
                          for i in range(n)]).T
    assert np.allclose(out["obs"][7], obs_fresh, atol=1e-12)
    assert np.all(b.episode == 3) and np.all(b.t_ep == 6)


def test_rollout_logp_and_noise(oracle):
    """a = mu + sigma eps with eps the env's action-stream normals at the
    global step; logp = sum of scipy's normal log-density of a."""
    stats = pytest.importorskip("scipy.stats")
    w = W.workload("ppo_65536", n_envs=4)
    m = oracle.model(w)
    n = 4
    ids = np.array([0, 1, 65535, 9])
    b = oracle.Batch(ids)
    oracle.reset(m, b)
    pw, vw = W.policy_weights(w, 0.05), W.value_weights(w, 0.05)
    t_g0 = 1000
    out = oracle.rollout(m, b, pw, vw, t_g0, 5)
    for t in range(5):
        head = oracle.mlp(pw, 18, 256, 16, True, out["obs"][t].T)
        val = oracle.mlp(vw, 18, 256, 1, True, out["obs"][t].T)
        assert np.allclose(out["value"][t], val[:, 0], atol=1e-12)
        mu = head[:, :8]
        ls = np.clip(head[:, 8:], w["logstd_min"], w["logstd_max"])
        for i in range(n):
            eps = oracle.normals(int(ids[i]), 0, t_g0 + t)
            a = out["act"][t, :, i]
            assert np.allclose(a, mu[i] + np.exp(ls[i]) * eps, atol=1e-12)
            lp = stats.norm.logpdf(a, loc=mu[i], scale=np.exp(ls[i])).sum()
            assert math.isclose(out["logp"][t, i], lp, rel_tol=1e-9, abs_tol=1e-9)


def test_rollout_matches_replay_of_its_own_actions(oracle):
    """The closed-loop rollout and an action replay of the actions it took
    produce the same rewards, dones and final state."""
    w = W.workload("dr_16384", episode_len=9)
    m = oracle.model(w)
    b1 = oracle.Batch(np.arange(5))
    oracle.reset(m, b1)
    b2 = b1.copy()
    out = oracle.rollout(m, b1, W.policy_weights(w), None, 0, 25)
    rew, done, _ = oracle.replay(m, b2, out["act"].astype(np.float32))
    # the replay path reads the actions rounded to float32
    assert np.array_equal(done, out["done"])
    assert np.allclose(rew, out["rew"], atol=1e-5)
    assert np.allclose(b1.state, b2.state, atol=1e-5)


@pytest.mark.parametrize("model", ["fossen", "paper"])
def test_logstd_clamp_pinned_beyond_both_bounds(oracle, model):
    """The log-std clamp of the policy head (A6: [-5, 2]).  The head's
    log-std rows are made constant by zero weights and biases of +50, -50,
    0.3 and -0.7: the clamp must give sigma = e^2, e^-5, e^0.3 and e^-0.7.
    Both the draw a - mu = sigma eps (normals pinned against cuRAND's words
    and Box-Muller's moments elsewhere) and the log-density, against
    scipy's normal logpdf at that sigma, are checked; a missing clamp
    (sigma = e^50), swapped bounds (every sigma = e^-5 or e^2) or a dropped
    term of the density fails.  The rollout's first step agrees with the
    same draw."""
    stats = pytest.importorskip("scipy.stats")
    paper = model == "paper"
    w = W.workload("paper_4096" if paper else "ppo_65536", n_envs=6)
    na = W.act_dim(w)
    d = W.obs_dim(w)
    pw = W.policy_weights(w, 0.1).astype(np.float32).copy()
    H = w["hidden"]
    o3 = H * d + H + H * H + H          # start of W3 [2 na][H]
    heads = np.array([50.0, -50.0, 0.3, -0.7, 50.0, -50.0, 0.3, -0.7][:na], dtype=np.float32)
    pw[o3 + na * H:o3 + 2 * na * H] = 0.0
    pw[o3 + 2 * na * H + na:o3 + 2 * na * H + 2 * na] = heads
    # the fp32 biases are the head's exact outputs (zero weights)
    sig = np.exp(np.clip(heads.astype(np.float64), -5.0, 2.0))
    assert np.allclose(np.log(sig), [2.0, -5.0, 0.3, -0.7, 2.0, -5.0, 0.3, -0.7][:na],
                       atol=1e-7)
    ids = np.array([0, 3, 17, 4095, 65535, 123456])
    obs = W.random_observations(9, len(ids), d)
    t_g = 77
    m = oracle.paper_model(w) if paper else oracle.model(w)
    act_fn = oracle.paper_policy_act if paper else oracle.policy_act
    act, logp = act_fn(m, pw, ids, t_g, obs.astype(np.float64))
    mu = oracle.mlp(pw, d, H, 2 * na, True, obs.astype(np.float64))[:, :na]
    for i, e in enumerate(ids):
        eps = oracle.normals(int(e), int(w["seed"]), t_g)[:na]
        assert np.allclose(act[i] - mu[i], sig * eps, rtol=1e-12, atol=1e-12)
        lp = stats.norm.logpdf(act[i], loc=mu[i], scale=sig).sum()
        assert math.isclose(logp[i], lp, rel_tol=1e-10, abs_tol=1e-9)
    # the rollout's step 0 takes the same draw from its own observation
    b = oracle.PaperBatch(ids) if paper else oracle.Batch(ids)
    (oracle.paper_reset if paper else oracle.reset)(m, b)
    roll = oracle.paper_rollout if paper else oracle.rollout
    out = roll(m, b, pw, None, t_g, 1, want=("obs", "act", "logp"))
    a0, lp0 = act_fn(m, pw, ids, t_g, out["obs"][0].T)
    assert np.allclose(out["act"][0].T, a0, rtol=1e-12, atol=1e-12)
    assert np.allclose(out["logp"][0], lp0, rtol=1e-12, atol=1e-12)
