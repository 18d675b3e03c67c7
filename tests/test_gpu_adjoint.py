"""GPU parity of the control-step adjoint (env_adjoint) against the oracle's
forward-mode dual numbers: for random directions (d_x0, d_a) the GPU's
<dJ/dx0, d_x0> + <dJ/da, d_a> equals the oracle's directional derivative of
the same window objective J = sum_t coef_t r_t + <lam_T, x_T>, per env;
unit directions check single components; windows with and without episode
ends, ragged env counts, the full-size window sampled, saturated thrusters,
the paper model (its adjoint state includes the action-history rows), and
argument rejection."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu

# |gpu - oracle| <= ADJ_TOL * sum_k |g_k d_k| per env: fp32 forward and
# adjoint arithmetic against the double dual-number derivative (measured
# 1.4e-7 .. 2.9e-7 over windows of 1 to 40 steps).
ADJ_TOL = 1e-5


def _setup(torch, n, T, warm, seed=0, **over):
    w = W.workload("ppo_65536", n_envs=n, w_vs=0.05, **over)
    env = make_env(w, policy=False)
    env.reset()
    if warm:
        acts = torch.from_numpy(W.replay_actions(seed + 1, warm, n, scale=0.8)).cuda()
        rew = torch.empty((warm, n), device="cuda")
        done = torch.empty((warm, n), dtype=torch.uint8, device="cuda")
        env.step_actions(acts, rew, done)
    rng = np.random.default_rng(seed)
    act = rng.uniform(-1.1, 1.1, (T, 8, n)).astype(np.float32)
    coef = (0.99 ** np.arange(T) * rng.uniform(0.5, 1.5)).astype(np.float32)
    lam_T = rng.normal(size=(13, n)).astype(np.float32)
    return w, env, act, coef, lam_T, rng


def _oracle_batch(oracle, env, ids):
    b = oracle.Batch(np.asarray(ids))
    b.state[:] = to_np(env.state)[:, ids]
    b.params[:] = to_np(env.params)[:, ids]
    b.t_ep[:] = to_np(env.t_ep)[ids]
    b.episode[:] = to_np(env.episode).view(np.uint32)[ids]
    return b


def _gpu_adjoint(torch, env, act, coef, lam_T):
    T, _, n = act.shape
    g = torch.empty((T, 8, n), device="cuda")
    l0 = torch.empty((13, n), device="cuda")
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    env.adjoint(torch.from_numpy(act).cuda(), torch.from_numpy(coef).cuda(), g,
                lam_T=torch.from_numpy(lam_T).cuda(), lam_0=l0, rew=rew, done=done)
    assert env.status().code == 0
    return to_np(g), to_np(l0), to_np(rew), to_np(done)


def _compare(oracle, m, b, act, coef, lam_T, g, l0, rng, ids, k_dirs=3, what=""):
    T = act.shape[0]
    n = len(ids)
    worst = 0.0
    for _ in range(k_dirs):
        ds0 = rng.normal(size=(13, n))
        da = rng.normal(size=(T, 8, n))
        _, dJ = oracle.adjoint_window(m, b, act[:, :, ids].astype(np.float64), coef,
                                      lam_T[:, ids], ds0, da)
        terms = g[:, :, ids] * da
        got = terms.sum(axis=(0, 1)) + (l0[:, ids] * ds0).sum(axis=0)
        scale = np.abs(terms).sum(axis=(0, 1)) + np.abs(l0[:, ids] * ds0).sum(axis=0)
        err = np.abs(got - dJ) / np.maximum(scale, 1e-6)
        worst = max(worst, float(err.max()))
    print(f"[adjoint {what}] max |<grad, d> - dJ| / sum|g d| = {worst:.3e} (tol {ADJ_TOL})")
    assert worst <= ADJ_TOL


@pytest.mark.parametrize("n,T,warm,L", [(300, 8, 5, 500),     # no episode end
                                        (257, 12, 4, 10),     # episode end at step 5
                                        (64, 1, 0, 500),      # single step from reset
                                        (130, 40, 3, 20)])    # long window, an end inside
def test_adjoint_matches_dual_numbers(oracle, n, T, warm, L):
    torch = need_gpu()
    w, env, act, coef, lam_T, rng = _setup(torch, n, T, warm, seed=n + T, episode_len=L)
    state0 = to_np(env.state).copy()
    g, l0, rew, done = _gpu_adjoint(torch, env, act, coef, lam_T)
    assert np.array_equal(to_np(env.state), state0)          # the env is not advanced
    m = oracle.model(w)
    ids = np.arange(n)
    b = _oracle_batch(oracle, env, ids)
    r_rew, r_done, _ = oracle.replay(m, b.copy(), act)
    assert np.array_equal(done, r_done)
    assert np.abs(rew - r_rew).max() <= 1e-4 * max(1.0, np.abs(r_rew).max())
    if L < warm + T:
        assert done.any()
    _compare(oracle, m, b, act, coef, lam_T, g, l0, rng, ids, what=f"n{n} T{T} L{L}")
    # saturated commands carry no gradient
    assert np.all(g[np.abs(act) > 1.0] == 0.0)


def test_adjoint_single_components(oracle):
    """Unit directions on three envs: every action component of every step
    and every initial-state component."""
    torch = need_gpu()
    n, T = 96, 4
    w, env, act, coef, lam_T, rng = _setup(torch, n, T, 6, seed=3)
    g, l0, _, _ = _gpu_adjoint(torch, env, act, coef, lam_T)
    m = oracle.model(w)
    ids = np.array([0, 47, 95])
    b = _oracle_batch(oracle, env, ids)
    a64 = act[:, :, ids].astype(np.float64)
    for c in range(13):
        ds0 = np.zeros((13, 3))
        ds0[c] = 1.0
        _, dJ = oracle.adjoint_window(m, b, a64, coef, lam_T[:, ids], ds0, np.zeros((T, 8, 3)))
        scale = np.abs(l0[:, ids]).max(axis=0)
        assert np.all(np.abs(l0[c, ids] - dJ) <= ADJ_TOL * 10 * np.maximum(scale, 1e-3)), c
    for t in range(T):
        for k in range(8):
            da = np.zeros((T, 8, 3))
            da[t, k] = 1.0
            _, dJ = oracle.adjoint_window(m, b, a64, coef, lam_T[:, ids], np.zeros((13, 3)), da)
            scale = np.abs(g[:, :, ids]).max(axis=(0, 1))
            assert np.all(np.abs(g[t, k, ids] - dJ) <= ADJ_TOL * 10 * np.maximum(scale, 1e-3)), (t, k)


def test_adjoint_full_size_sampled(oracle):
    """The bench's window: 65,536 envs x 32 steps, episode ends inside for
    every env; 64 sampled envs against the oracle."""
    torch = need_gpu()
    n, T = 65536, 32
    w, env, act, coef, lam_T, rng = _setup(torch, n, T, 2, seed=9, episode_len=20)
    g, l0, rew, done = _gpu_adjoint(torch, env, act, coef, lam_T)
    assert done[17].all() and not done[:17].any()
    ids = np.unique(np.r_[0, 1, 127, 128, n - 1, rng.integers(0, n, 59)])
    m = oracle.model(w)
    b = _oracle_batch(oracle, env, ids)
    _compare(oracle, m, b, act, coef, lam_T, g, l0, rng, ids, k_dirs=2, what="65536 x 32")
    # before the episode end nothing reaches the terminal term or later rewards
    assert np.all(np.isfinite(g)) and np.all(np.isfinite(l0))


def test_adjoint_rejects_bad_arguments():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n = 64
    env = make_env(W.workload("ppo_65536", n_envs=n), policy=False)
    env.reset()
    g = torch.empty((65, 8, n), device="cuda")
    act = torch.zeros((65, 8, n), device="cuda")
    coef = torch.ones(65, device="cuda")
    with pytest.raises(auvenv.AuvError) as ei:
        env.adjoint(act, coef, g)                               # T = 65
    assert ei.value.code == auvenv.AUV_ERR_INVALID
    with pytest.raises(auvenv.AuvError) as ei:
        env.adjoint(act[:4].cpu(), coef[:4], g[:4])             # host actions
    assert ei.value.code == auvenv.AUV_ERR_SIZE
    env16 = make_env(W.workload("ppo_65536", n_envs=n, substeps=16), policy=False)
    with pytest.raises(auvenv.AuvError) as ei:
        env16.adjoint(act[:4], coef[:4], g[:4])
    assert ei.value.code == auvenv.AUV_ERR_UNSUPPORTED


@pytest.mark.parametrize("n,T,L,K", [(300, 10, 500, 4), (129, 12, 9, 3), (64, 6, 500, 8)])
def test_paper_adjoint_matches_dual_numbers(oracle, n, T, L, K):
    """The paper model: 61 adjoint rows (p, q, nu, the 8 x 6 history), the
    moving-average term carrying gradient from later rewards to earlier
    actions, episode ends inside the window."""
    torch = need_gpu()
    w = W.workload("paper_tiny", n_envs=n, substeps=4, dr_enable=1, mavg_len=K, g_eff=0.05,
                   episode_len=L)
    env = make_env(w, policy=False)
    env.reset()
    warm = torch.from_numpy(W.replay_actions(n + 1, 5, n, scale=0.8, act=6)).cuda()
    env.step_actions(warm, torch.empty((5, n), device="cuda"),
                     torch.empty((5, n), dtype=torch.uint8, device="cuda"))
    rng = np.random.default_rng(n + T)
    act = rng.uniform(-1.1, 1.1, (T, 6, n)).astype(np.float32)
    coef = (0.99 ** np.arange(T)).astype(np.float32)
    lam_T = rng.normal(size=(61, n)).astype(np.float32)
    st0 = to_np(env.state).copy()
    g = torch.empty((T, 6, n), device="cuda")
    l0 = torch.empty((61, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    env.adjoint(torch.from_numpy(act).cuda(), torch.from_numpy(coef).cuda(), g,
                lam_T=torch.from_numpy(lam_T).cuda(), lam_0=l0, done=done)
    assert env.status().code == 0
    assert np.array_equal(to_np(env.state), st0)
    if L < 5 + T:
        assert to_np(done).any()
    m = oracle.paper_model(w)
    b = oracle.PaperBatch(np.arange(n))
    b.state[:] = st0
    b.params[:] = to_np(env.params)
    b.t_ep[:] = to_np(env.t_ep)
    b.episode[:] = to_np(env.episode).view(np.uint32)
    G, L0 = to_np(g), to_np(l0)
    worst = 0.0
    for _ in range(3):
        ds0 = rng.normal(size=(61, n))
        da = rng.normal(size=(T, 6, n))
        _, dJ = oracle.paper_adjoint_window(m, b, act.astype(np.float64), coef, lam_T, ds0, da)
        terms = G * da
        got = terms.sum(axis=(0, 1)) + (L0 * ds0).sum(axis=0)
        scale = np.abs(terms).sum(axis=(0, 1)) + np.abs(L0 * ds0).sum(axis=0)
        worst = max(worst, float((np.abs(got - dJ) / np.maximum(scale, 1e-6)).max()))
    print(f"[paper adjoint n{n} T{T} L{L} K{K}] {worst:.3e} (tol {ADJ_TOL})")
    assert worst <= ADJ_TOL
    assert np.all(G[np.abs(act) > 1.0] == 0.0)
