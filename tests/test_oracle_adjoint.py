"""Pins for the oracle of the adjoint kernels: the directional derivative of
an action-replay window objective J = sum_t coef_t r_t + <lam_T, x_T>
computed by forward-mode dual numbers over the model code (oracle
adjoint_window) against central differences of the same J in double, a
one-substep closed form, linearity in the direction, the gradient cut at an
episode end, and zero derivative through clipped thruster commands.  The
closed-loop window of SHAC (policy network inside, terminal critic): its
value equals the oracle's own rollout, its weight derivative matches central
differences, and the critic term alone is linear in the direction."""
import numpy as np
import pytest

from oracle import oracle as O
from paper_2512_13359_gb300 import workloads as W


def _setup(n=6, T=5, seed=0, warm=7, **over):
    """A batch moved off its reset state by `warm` replay steps (so that
    velocities, angular rates and the current are all non-zero), and
    actions for the window away from the clip edges."""
    w = W.workload("ppo_65536", n_envs=n, w_vs=0.05, **over)
    m = O.model(w)
    b = O.Batch(np.arange(n) + 11)
    O.reset(m, b)
    rng = np.random.default_rng(seed)
    if warm:
        O.replay(m, b, W.replay_actions(seed + 1, warm, n, scale=0.8))
    act = rng.uniform(-0.95, 0.95, (T, 8, n))
    return w, m, b, act, rng


def _dirs(rng, T, n):
    return rng.normal(size=(13, n)), rng.normal(size=(T, 8, n))


def _shifted(b, act, ds0, da, h):
    b2 = b.copy()
    b2.state[0:13] = b.state[0:13] + h * ds0
    return b2, act + h * da


def test_dual_derivative_matches_central_differences():
    T, n = 6, 5
    w, m, b, act, rng = _setup(n=n, T=T)
    coef = rng.normal(size=T)
    lam = rng.normal(size=(13, n))
    ds0, da = _dirs(rng, T, n)
    zero0, zeroa = np.zeros((13, n)), np.zeros((T, 8, n))
    J, dJ = O.adjoint_window(m, b, act, coef, lam, ds0, da)
    h = 1e-6
    bp, ap = _shifted(b, act, ds0, da, h)
    bm, am = _shifted(b, act, ds0, da, -h)
    Jp, _ = O.adjoint_window(m, bp, ap, coef, lam, zero0, zeroa)
    Jm, _ = O.adjoint_window(m, bm, am, coef, lam, zero0, zeroa)
    fd = (Jp - Jm) / (2 * h)
    assert np.all(np.abs(dJ) > 1e-3)
    assert np.allclose(dJ, fd, rtol=1e-6, atol=1e-9), (dJ, fd)
    # the window leaves the batch untouched
    J2, _ = O.adjoint_window(m, b, act, coef, lam, zero0, zeroa)
    assert np.array_equal(J, J2)


def test_one_substep_from_rest_closed_form():
    """From rest, with no current, no buoyancy offset and the centre of
    buoyancy at the origin, one substep gives nu' = h M^-1 tau and
    p' = p + h R(q) v', so that for lam_T on (p, nu) and coef = 0
    dJ/da_j = sum_k lam_nu,k h B_kj / M_k + lam_p . h R(q) (h B_vj / M_v)
    with B = alloc * thrust_max."""
    n, T = 4, 1
    w, m, b, act, rng = _setup(n=n, T=T, warm=0, substeps=1, dr_enable=0, current_range=0.0)
    assert np.all(b.state[7:13] == 0) and np.all(b.params[10:17] == 0)
    lam = np.zeros((13, n))
    lam[0:3] = rng.normal(size=(3, n))
    lam[7:13] = rng.normal(size=(6, n))
    h = float(w["dt"])
    Minv = 1.0 / (np.r_[[w["mass"]] * 3, w["inertia"]] + np.asarray(w["added_mass"]))
    Bm = np.asarray(w["alloc"], dtype=np.float64).reshape(6, 8) * w["thrust_max"]
    for j in range(8):
        da = np.zeros((T, 8, n))
        da[0, j] = 1.0
        _, dJ = O.adjoint_window(m, b, act, np.zeros(T), lam, np.zeros((13, n)), da)
        for i in range(n):
            q = b.state[3:7, i]
            wq, x, y, z = q
            R = np.array([[1 - 2 * (y * y + z * z), 2 * (x * y - wq * z), 2 * (x * z + wq * y)],
                          [2 * (x * y + wq * z), 1 - 2 * (x * x + z * z), 2 * (y * z - wq * x)],
                          [2 * (x * z - wq * y), 2 * (y * z + wq * x), 1 - 2 * (x * x + y * y)]])
            dnu = h * Minv * Bm[:, j]
            want = lam[7:13, i] @ dnu + lam[0:3, i] @ (h * R @ dnu[0:3])
            assert dJ[i] == pytest.approx(want, rel=1e-12, abs=1e-15)


def test_derivative_is_linear_in_the_direction():
    T, n = 4, 3
    w, m, b, act, rng = _setup(n=n, T=T, seed=3)
    coef, lam = rng.normal(size=T), rng.normal(size=(13, n))
    s1, a1 = _dirs(rng, T, n)
    s2, a2 = _dirs(rng, T, n)
    _, d1 = O.adjoint_window(m, b, act, coef, lam, s1, a1)
    _, d2 = O.adjoint_window(m, b, act, coef, lam, s2, a2)
    _, d12 = O.adjoint_window(m, b, act, coef, lam, s1 + 2 * s2, a1 + 2 * a2)
    assert np.allclose(d12, d1 + 2 * d2, rtol=1e-12, atol=1e-14)


def test_episode_end_cuts_the_gradient():
    """With the episode ending at window step 2, nothing before or at that
    step (actions 0..2, the initial state) reaches rewards of steps 3.. or
    the terminal state; actions after it do."""
    T, n = 6, 4
    w, m, b, act, rng = _setup(n=n, T=T, warm=0, episode_len=3)
    coef = np.r_[0.0, 0.0, 0.0, rng.normal(size=3)]
    lam = rng.normal(size=(13, n))
    ds0, da = _dirs(rng, T, n)
    da_before = da.copy()
    da_before[3:] = 0
    _, dJ = O.adjoint_window(m, b, act, coef, lam, ds0, da_before)
    assert np.all(dJ == 0.0)
    da_after = da.copy()
    da_after[:3] = 0
    _, dJ = O.adjoint_window(m, b, act, coef, lam, np.zeros((13, n)), da_after)
    assert np.all(np.abs(dJ) > 0)


def test_clipped_commands_have_zero_derivative():
    T, n = 3, 4
    w, m, b, act, rng = _setup(n=n, T=T, seed=5)
    act[:, 2] = 1.4          # thruster 2 saturated high at every step
    act[:, 5] = -1.7         # thruster 5 saturated low
    coef, lam = rng.normal(size=T), rng.normal(size=(13, n))
    da = np.zeros((T, 8, n))
    da[:, 2] = rng.normal(size=(T, n))
    da[:, 5] = rng.normal(size=(T, n))
    _, dJ = O.adjoint_window(m, b, act, coef, lam, np.zeros((13, n)), da)
    assert np.all(dJ == 0.0)


# ---------------------------------------------------------------------------
# Closed loop (SHAC's window with the policy network and a terminal critic)
# ---------------------------------------------------------------------------
def _smooth_policy(w, scale_mu=0.15, ls_bias=-3.0):
    """Policy weights whose actions stay inside the thrusters' range (small
    mean, sigma = e^-3), so the window objective is smooth in the weights."""
    pw = W.policy_weights(w).astype(np.float64)
    H = w["hidden"]
    o3 = H * 18 + H + H * H + H
    W3 = pw[o3:o3 + 16 * H].reshape(16, H)
    W3[:8] *= scale_mu
    W3[8:] *= 0.1
    pw[o3 + 16 * H + 8:o3 + 16 * H + 16] = ls_bias
    return pw.astype(np.float32)


def _closed_loop_setup(n=4, T=5, seed=0, **over):
    w = W.workload("ppo_65536", n_envs=n, hidden=16, w_vs=0.05, mlp="fp32", **over)
    m = O.model(w)
    b = O.Batch(np.arange(n) + 3)
    O.reset(m, b)
    O.replay(m, b, W.replay_actions(seed + 1, 4, n, scale=0.8))
    return w, m, b


def test_shac_window_value_equals_the_rollout():
    T, n = 6, 4
    w, m, b = _closed_loop_setup(n, T)
    pw = W.policy_weights(w)
    coef = np.random.default_rng(1).uniform(0.5, 1.5, T)
    J, _ = O.shac_window(m, b, pw, None, None, 100, T, coef, 0.0)
    ref = O.rollout(m, b.copy(), pw, None, 100, T, want=("rew",))
    assert np.allclose(J, coef @ ref["rew"], rtol=1e-12, atol=1e-12)


def test_shac_window_derivative_matches_central_differences():
    T, n = 5, 3
    w, m, b = _closed_loop_setup(n, T, seed=2)
    pw = _smooth_policy(w)
    vw = W.value_weights(w, 0.1)
    rng = np.random.default_rng(3)
    coef = rng.uniform(0.5, 1.5, T)
    d = rng.normal(size=pw.size) * np.abs(pw).mean()
    J, dJ = O.shac_window(m, b, pw, d, vw, 7, T, coef, 0.7)
    h = 2e-3
    Jp, _ = O.shac_window(m, b, (pw + h * d).astype(np.float32), None, vw, 7, T, coef, 0.7)
    Jm, _ = O.shac_window(m, b, (pw - h * d).astype(np.float32), None, vw, 7, T, coef, 0.7)
    fd = (Jp - Jm) / (2 * h)
    assert np.all(np.abs(dJ) > 1e-4)
    # the perturbed weights are rounded to float32 (the oracle's weight type):
    # that noise, ~1e-5 of the largest derivative here, bounds the agreement
    assert np.all(np.abs(dJ - fd) <= 3e-4 * np.abs(fd) + 3e-5 * np.abs(fd).max()), (dJ, fd)


def test_shac_terminal_critic_alone():
    """With coef = 0 only the critic term reaches the weights (through the
    final state); its derivative is linear in the direction."""
    T, n = 4, 3
    w, m, b = _closed_loop_setup(n, T, seed=4)
    pw = _smooth_policy(w)
    vw = W.value_weights(w, 0.1)
    rng = np.random.default_rng(5)
    d1, d2 = rng.normal(size=pw.size), rng.normal(size=pw.size)
    _, a = O.shac_window(m, b, pw, d1, vw, 0, T, np.zeros(T), 1.0)
    _, c = O.shac_window(m, b, pw, d2, vw, 0, T, np.zeros(T), 1.0)
    _, ac = O.shac_window(m, b, pw, d1 - 3 * d2, vw, 0, T, np.zeros(T), 1.0)
    assert np.all(np.abs(a) > 0)
    assert np.allclose(ac, a - 3 * c, rtol=1e-10, atol=1e-14)
    _, z = O.shac_window(m, b, pw, d1, None, 0, T, np.zeros(T), 1.0)
    assert np.all(z == 0.0)


# ---------------------------------------------------------------------------
# The paper model's window (state with the action history)
# ---------------------------------------------------------------------------
def _paper_setup(n=5, T=6, seed=0, warm=5, **over):
    w = W.workload("paper_tiny", n_envs=n, substeps=4, dr_enable=1, mavg_len=4,
                   g_eff=0.05, **over)
    m = O.paper_model(w)
    b = O.PaperBatch(np.arange(n) + 7)
    O.paper_reset(m, b)
    if warm:
        O.paper_replay(m, b, W.replay_actions(seed + 1, warm, n, scale=0.8, act=6))
    rng = np.random.default_rng(seed)
    act = rng.uniform(-0.95, 0.95, (T, 6, n))
    return w, m, b, act, rng


def test_paper_window_derivative_matches_central_differences():
    """Directions on every state row, the history slots included, and on
    the actions; the history makes an action reach later rewards."""
    T, n = 7, 4
    w, m, b, act, rng = _paper_setup(n, T)
    assert np.abs(b.state[13:37]).max() > 0            # K = 4 slots filled
    coef = rng.normal(size=T)
    lam = rng.normal(size=(61, n))
    ds0, da = rng.normal(size=(61, n)), rng.normal(size=(T, 6, n))
    J, dJ = O.paper_adjoint_window(m, b, act, coef, lam, ds0, da)
    h = 1e-6
    bp, bm = b.copy(), b.copy()
    bp.state[:] = b.state + h * ds0
    bm.state[:] = b.state - h * ds0
    z0, za = np.zeros((61, n)), np.zeros((T, 6, n))
    Jp, _ = O.paper_adjoint_window(m, bp, act + h * da, coef, lam, z0, za)
    Jm, _ = O.paper_adjoint_window(m, bm, act - h * da, coef, lam, z0, za)
    fd = (Jp - Jm) / (2 * h)
    assert np.all(np.abs(dJ) > 1e-3)
    assert np.allclose(dJ, fd, rtol=1e-6, atol=1e-9), (dJ, fd)


def test_paper_action_reaches_later_rewards_through_the_history():
    """With coef only on the last step and no terminal term, the first
    action still has a derivative (through the moving-average term of the
    later reward), which vanishes with w_mavg = 0."""
    T, n = 3, 3
    w, m, b, act, rng = _paper_setup(n, T, seed=2)
    coef = np.array([0.0, 0.0, 1.0])
    da = np.zeros((T, 6, n))
    da[0] = rng.normal(size=(6, n))
    # the first action also moves the state, so isolate the history path by
    # comparing against the same derivative without the moving-average term
    _, with_hist = O.paper_adjoint_window(m, b, act, coef, None, np.zeros((61, n)), da)
    m0 = O.paper_model(dict(w, w_mavg=0.0))
    _, without = O.paper_adjoint_window(m0, b, act, coef, None, np.zeros((61, n)), da)
    assert np.all(np.abs(with_hist - without) > 1e-8)


def test_paper_shac_window_value_and_derivative():
    """The paper model's closed-loop window: its value equals the oracle's
    own paper rollout, and its weight derivative matches central differences
    (smooth policy: small means, sigma = e^-3)."""
    T, n, H = 5, 3, 16
    w = W.workload("paper_tiny", n_envs=n, hidden=H, policy_out=12, mlp="fp32", mavg_len=3,
                   substeps=2)
    m = O.paper_model(w)
    b = O.PaperBatch(np.arange(n) + 5)
    O.paper_reset(m, b)
    O.paper_replay(m, b, W.replay_actions(3, 4, n, scale=0.8, act=6))
    pw = W.policy_weights(w).astype(np.float64)
    o3 = H * 12 + H + H * H + H
    W3 = pw[o3:o3 + 12 * H].reshape(12, H)
    W3[:6] *= 0.15
    W3[6:] *= 0.1
    pw[o3 + 12 * H + 6:o3 + 12 * H + 12] = -3.0
    pw = pw.astype(np.float32)
    coef = np.random.default_rng(4).uniform(0.5, 1.5, T)
    J, _ = O.paper_shac_window(m, b, pw, None, None, 50, T, coef, 0.0)
    ref = O.paper_rollout(m, b.copy(), pw, None, 50, T)
    assert np.allclose(J, coef @ ref["rew"], rtol=1e-12, atol=1e-12)
    vw = W.value_weights(w, 0.1)
    d = np.random.default_rng(5).normal(size=pw.size) * np.abs(pw).mean()
    _, dJ = O.paper_shac_window(m, b, pw, d, vw, 50, T, coef, 0.7)
    h = 2e-3
    Jp, _ = O.paper_shac_window(m, b, (pw + h * d).astype(np.float32), None, vw, 50, T, coef, 0.7)
    Jm, _ = O.paper_shac_window(m, b, (pw - h * d).astype(np.float32), None, vw, 50, T, coef, 0.7)
    fd = (Jp - Jm) / (2 * h)
    assert np.all(np.abs(dJ) > 1e-5)
    assert np.all(np.abs(dJ - fd) <= 3e-4 * np.abs(fd) + 3e-5 * np.abs(fd).max()), (dJ, fd)
