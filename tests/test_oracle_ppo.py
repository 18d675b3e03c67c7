"""Pins for the oracle's generalised advantage estimation against
formulations that do not share its recursion: the lambda = 1 case is the
discounted Monte-Carlo return minus the value (summed explicitly per
episode), lambda = 0 is the one-step TD error, the general case equals the
lambda-weighted sum of n-step advantages (the definition GAE is derived
from), and a 3-step example computed by hand."""
import numpy as np
import pytest

from oracle import ppo_oracle as P


def _episode_data(seed, T, n, p_done=0.1):
    rng = np.random.default_rng(seed)
    rew = rng.normal(size=(T, n))
    value = rng.normal(size=(T, n))
    done = (rng.random((T, n)) < p_done).astype(np.uint8)
    last = rng.normal(size=n)
    return rew, done, value, last


def _discounted_to_end(rew, done, value, last, gamma, t, i):
    """sum_{k>=t} gamma^{k-t} r_k up to the episode end, plus the bootstrap
    gamma^{T-t} V_T when the trajectory ends inside the episode."""
    T = rew.shape[0]
    g, disc = 0.0, 1.0
    for k in range(t, T):
        g += disc * rew[k, i]
        if done[k, i]:
            return g
        disc *= gamma
    return g + disc * last[i]


def test_lambda_one_is_monte_carlo_return():
    rew, done, value, last = _episode_data(1, 25, 7)
    gamma = 0.97
    adv, ret = P.gae(rew, done, value, last, gamma, 1.0)
    for t in range(25):
        for i in range(7):
            mc = _discounted_to_end(rew, done, value, last, gamma, t, i)
            assert ret[t, i] == pytest.approx(mc, rel=1e-12, abs=1e-12)
            assert adv[t, i] == pytest.approx(mc - value[t, i], rel=1e-12, abs=1e-12)


def test_lambda_zero_is_td_error():
    rew, done, value, last = _episode_data(2, 20, 5)
    gamma = 0.9
    adv, _ = P.gae(rew, done, value, last, gamma, 0.0)
    v_next = np.vstack([value[1:], last[None]])
    assert np.allclose(adv, rew + gamma * (1 - done) * v_next - value, rtol=1e-14, atol=1e-14)


def test_general_lambda_is_weighted_n_step_sum():
    """A_t = (1 - lam) sum_{n>=1} lam^{n-1} A_t^(n) with the n-step
    advantages A^(n) = sum_{k<n} gamma^k r_{t+k} + gamma^n V_{t+n} - V_t,
    truncated at the trajectory end (the tail weight lam^{N-1} goes to the
    longest advantage) and at episode ends."""
    T, n_env, gamma, lam = 12, 4, 0.95, 0.8
    rew, done, value, last = _episode_data(3, T, n_env, p_done=0.15)
    adv, _ = P.gae(rew, done, value, last, gamma, lam)
    vals = np.vstack([value, last[None]])
    for i in range(n_env):
        for t in range(T):
            # steps available in this episode from t (inclusive of a done step)
            L = 0
            while t + L < T:
                L += 1
                if done[t + L - 1, i]:
                    break
            terminal = bool(done[t + L - 1, i])
            adv_n = []
            for m in range(1, L + 1):
                g = sum(gamma ** k * rew[t + k, i] for k in range(m))
                boot = 0.0 if (terminal and m == L) else gamma ** m * vals[t + m, i]
                adv_n.append(g + boot - value[t, i])
            w = [(1 - lam) * lam ** (m - 1) for m in range(1, L)] + [lam ** (L - 1)]
            assert adv[t, i] == pytest.approx(np.dot(w, adv_n), rel=1e-11, abs=1e-12)


def test_hand_computed_three_steps():
    rew = np.array([[1.0], [2.0], [3.0]])
    value = np.array([[0.5], [0.25], [1.0]])
    done = np.array([[0], [1], [0]], dtype=np.uint8)
    last = np.array([2.0])
    g, l = 0.5, 0.5
    # t = 2: delta = 3 + 0.5 * 2 - 1 = 3; A = 3
    # t = 1 (done): delta = 2 - 0.25 = 1.75; A = 1.75
    # t = 0: delta = 1 + 0.5 * 0.25 - 0.5 = 0.625; A = 0.625 + 0.25 * 1.75 = 1.0625
    adv, ret = P.gae(rew, done, value, last, g, l)
    assert np.allclose(adv[:, 0], [1.0625, 1.75, 3.0], rtol=0, atol=1e-15)
    assert np.allclose(ret[:, 0], [1.5625, 2.0, 4.0], rtol=0, atol=1e-15)
