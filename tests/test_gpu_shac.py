"""GPU parity of SHAC's closed-loop window (env_shac_window) against the
oracle's dual-number window: each env's objective J, and the policy
gradient projected on random weight directions (<grad, d> against the sum
over envs of the oracle's directional derivatives), for a smooth policy and
one whose commands saturate, with and without episode ends inside the
window and with and without the terminal critic; the env's advance and
rejections."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu

# |<grad, d> - sum_i dJ_i| <= SHAC_TOL * sum_k |grad_k d_k|: fp32 windows
# (forward, cuBLAS fp32 GEMMs, VJPs) against the double dual numbers
# (measured 1.6e-9 .. 1.3e-8).  Single coordinates: within COORD_TOL of the
# largest gradient component.
SHAC_TOL = 1e-6
COORD_TOL = 1e-4


def _smooth(pw, H):
    pw = pw.astype(np.float64).copy()
    o3 = H * 18 + H + H * H + H
    W3 = pw[o3:o3 + 16 * H].reshape(16, H)
    W3[:8] *= 0.15
    W3[8:] *= 0.1
    pw[o3 + 16 * H + 8:o3 + 16 * H + 16] = -3.0
    return pw.astype(np.float32)


def _window(torch, oracle, n, T, H, L, smooth, critic, seed):
    w = W.workload("ppo_65536", n_envs=n, hidden=H, mlp="fp32", w_vs=0.05, episode_len=L)
    env = make_env(w, policy=False)
    env.reset()
    warm = torch.from_numpy(W.replay_actions(seed, 3, n, scale=0.8)).cuda()
    env.step_actions(warm, torch.empty((3, n), device="cuda"),
                     torch.empty((3, n), dtype=torch.uint8, device="cuda"))
    pw = W.policy_weights(w, 0.05)
    if smooth:
        pw = _smooth(pw, H)
    vw = W.value_weights(w, 0.1) if critic else None
    rng = np.random.default_rng(seed)
    coef = (0.99 ** np.arange(T) * rng.uniform(0.5, 1.5) / n).astype(np.float32)
    coef_V = 0.8 / n
    b = oracle.Batch(np.arange(n))
    b.state[:] = to_np(env.state)
    b.params[:] = to_np(env.params)
    b.t_ep[:] = to_np(env.t_ep)
    b.episode[:] = to_np(env.episode).view(np.uint32)
    t_g0 = env.t_g
    grad = torch.empty(pw.size, device="cuda")
    J = torch.empty(n, device="cuda")
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    env.shac_window(torch.from_numpy(pw).cuda(), None if vw is None else torch.from_numpy(vw).cuda(),
                    torch.from_numpy(coef).cuda(), coef_V, grad, J=J, rew=rew, done=done)
    assert env.status().code == 0
    assert env.t_g == t_g0 + T
    return w, env, b, pw, vw, coef, coef_V, t_g0, to_np(grad), to_np(J), to_np(rew), to_np(done), rng


def _check(oracle, w, b, pw, vw, coef, coef_V, t_g0, T, grad, J, rng, k_dirs=3, what=""):
    m = oracle.model(w)
    worst = 0.0
    for k in range(k_dirs):
        d = rng.normal(size=pw.size)
        Jr, dJ = oracle.shac_window(m, b, pw, d, vw, t_g0, T, coef, coef_V)
        if k == 0:
            assert np.abs(J - Jr).max() <= 1e-4 * max(np.abs(Jr).max(), 1e-6), "J"
        got = float(grad.astype(np.float64) @ d)
        scale = float(np.abs(grad.astype(np.float64) * d).sum())
        worst = max(worst, abs(got - dJ.sum()) / scale)
    print(f"[shac {what}] |<grad, d> - dJ| / sum|grad d| = {worst:.3e} (tol {SHAC_TOL})")
    assert worst <= SHAC_TOL


@pytest.mark.parametrize("n,T,L,smooth,critic", [
    (64, 6, 500, True, True),        # smooth policy, no episode end, critic
    (100, 8, 5, False, True),        # saturating commands, an end at step 1
    (37, 4, 500, False, False),      # no critic
    (130, 12, 9, True, True)])       # an end inside a longer window
def test_shac_window_matches_dual_numbers(oracle, n, T, L, smooth, critic):
    torch = need_gpu()
    out = _window(torch, oracle, n, T, 64, L, smooth, critic, seed=n + T)
    w, env, b, pw, vw, coef, coef_V, t_g0, grad, J, rew, done, rng = out
    if L < 3 + T:
        assert done.any()
    _check(oracle, w, b, pw, vw, coef, coef_V, t_g0, T, grad, J, rng,
           what=f"n{n} T{T} L{L} smooth={smooth} critic={critic}")
    # single weights of every layer: W1, b1, W2, b2, W3 (mean and log-std
    # rows), b3 (mean and log-std)
    H = 64
    o = dict(W1=5, b1=18 * H + 3, W2=18 * H + H + 777, b2=18 * H + H + H * H + 9)
    o3 = 18 * H + H + H * H + H
    o.update(W3mu=o3 + 2 * H + 7, W3ls=o3 + 11 * H + 5, b3mu=o3 + 16 * H + 1,
             b3ls=o3 + 16 * H + 12)
    m = oracle.model(w)
    top = np.abs(grad).max()
    for name, k in o.items():
        d = np.zeros(pw.size)
        d[k] = 1.0
        _, dJ = oracle.shac_window(m, b, pw, d, vw, t_g0, T, coef, coef_V)
        assert abs(grad[k] - dJ.sum()) <= COORD_TOL * top, (name, grad[k], dJ.sum())


def test_shac_window_hidden_256_long_window(oracle):
    """The rollout's network width and SHAC's usual horizon: 512 envs x 32
    steps, hidden 256, one direction."""
    torch = need_gpu()
    out = _window(torch, oracle, 512, 32, 256, 20, True, True, seed=5)
    w, env, b, pw, vw, coef, coef_V, t_g0, grad, J, rew, done, rng = out
    assert done[16].all()
    _check(oracle, w, b, pw, vw, coef, coef_V, t_g0, 32, grad, J, rng, k_dirs=1,
           what="512 x 32, hidden 256")


def test_shac_window_advances_like_a_replay(oracle):
    """After the window the env's state equals the oracle's closed-loop
    rollout of the same policy from the same state; rewards and dones too."""
    torch = need_gpu()
    n, T = 200, 7
    out = _window(torch, oracle, n, T, 64, 6, False, False, seed=11)
    w, env, b, pw, vw, coef, coef_V, t_g0, grad, J, rew, done, rng = out
    m = oracle.model(w)
    ref = oracle.rollout(m, b, pw, None, t_g0, T, want=("rew",))
    assert np.array_equal(done, ref["done"])
    assert np.abs(rew - ref["rew"]).max() <= 1e-4 * max(1.0, np.abs(ref["rew"]).max())
    st = to_np(env.state)
    assert np.abs(st[:13] - b.state[:13]).max() <= 1e-4


@pytest.mark.parametrize("n,T,L,smooth", [(100, 6, 500, True), (130, 10, 7, False)])
def test_paper_shac_window_matches_dual_numbers(oracle, n, T, L, smooth):
    """The paper model in closed loop: policy 12 -> 64 -> 64 -> 12, the
    critic, the 61-row adjoint with the action history, episode ends."""
    torch = need_gpu()
    H = 64
    w = W.workload("paper_tiny", n_envs=n, hidden=H, policy_out=12, mlp="fp32", mavg_len=3,
                   substeps=4, dr_enable=1, g_eff=0.05, episode_len=L)
    env = make_env(w, policy=False)
    env.reset()
    warm = torch.from_numpy(W.replay_actions(n, 3, n, scale=0.8, act=6)).cuda()
    env.step_actions(warm, torch.empty((3, n), device="cuda"),
                     torch.empty((3, n), dtype=torch.uint8, device="cuda"))
    pw = W.policy_weights(w, 0.05).astype(np.float64)
    if smooth:
        o3 = H * 12 + H + H * H + H
        W3 = pw[o3:o3 + 12 * H].reshape(12, H)
        W3[:6] *= 0.15
        W3[6:] *= 0.1
        pw[o3 + 12 * H + 6:o3 + 12 * H + 12] = -3.0
    pw = pw.astype(np.float32)
    vw = W.value_weights(w, 0.1)
    b = oracle.PaperBatch(np.arange(n))
    b.state[:] = to_np(env.state)
    b.params[:] = to_np(env.params)
    b.t_ep[:] = to_np(env.t_ep)
    b.episode[:] = to_np(env.episode).view(np.uint32)
    t_g0 = env.t_g
    coef = (0.99 ** np.arange(T) / n).astype(np.float32)
    grad = torch.empty(pw.size, device="cuda")
    J = torch.empty(n, device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    env.shac_window(torch.from_numpy(pw).cuda(), torch.from_numpy(vw).cuda(),
                    torch.from_numpy(coef).cuda(), 0.6 / n, grad, J=J, done=done)
    assert env.status().code == 0
    if L < 3 + T:
        assert to_np(done).any()
    m = oracle.paper_model(w)
    g = to_np(grad).astype(np.float64)
    rng = np.random.default_rng(n)
    worst = 0.0
    for k in range(3):
        d = rng.normal(size=pw.size)
        Jr, dJ = oracle.paper_shac_window(m, b, pw, d, vw, t_g0, T, coef, 0.6 / n)
        if k == 0:
            assert np.abs(to_np(J) - Jr).max() <= 1e-4 * max(np.abs(Jr).max(), 1e-6)
        worst = max(worst, abs(g @ d - dJ.sum()) / np.abs(g * d).sum())
    print(f"[paper shac n{n} T{T} L{L} smooth={smooth}] {worst:.3e} (tol {SHAC_TOL})")
    assert worst <= SHAC_TOL
    ref = oracle.paper_rollout(m, b, pw, None, t_g0, T, want=("rew",))
    assert np.array_equal(to_np(done), ref["done"])
    assert np.abs(to_np(env.state)[:13] - b.state[:13]).max() <= 1e-4
    assert np.abs(to_np(env.state)[13:] - b.state[13:]).max() <= 1e-6


def test_shac_window_rejects_bad_arguments():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n = 64
    w = W.workload("ppo_65536", n_envs=n, hidden=64, mlp="fp32")
    env = make_env(w, policy=False)
    env.reset()
    pw = torch.from_numpy(W.policy_weights(w)).cuda()
    g = torch.empty_like(pw)
    coef = torch.ones(65, device="cuda")
    with pytest.raises(auvenv.AuvError) as ei:
        env.shac_window(pw, None, coef, 0.0, g)                  # T = 65
    assert ei.value.code == auvenv.AUV_ERR_INVALID
    with pytest.raises(auvenv.AuvError) as ei:
        env.shac_window(pw.cpu(), None, coef[:4], 0.0, g)        # host weights
    assert ei.value.code == auvenv.AUV_ERR_SIZE


def test_shac_critic_targets_and_regression(oracle):
    """SHAC's critic step from the window's outputs: the observations the
    window returns (the rollout's layout) equal the oracle's closed-loop
    rollout's, the TD(lambda) targets are env_gae's returns over the
    window's rewards, dones and critic values (bootstrap at the final
    observation), and the value-only learner's gradient on (obs, targets)
    matches the oracle's critic regression."""
    torch = need_gpu()
    from oracle import ppo_oracle as P
    from paper_2512_13359_gb300 import auvenv
    n, T, H = 256, 8, 64
    w = W.workload("ppo_65536", n_envs=n, hidden=H, mlp="fp32", has_value=1, episode_len=6)
    env = make_env(w)                       # the env's own value network is the critic
    env.reset()
    b = oracle.Batch(np.arange(n))
    b.state[:] = to_np(env.state)
    b.params[:] = to_np(env.params)
    b.t_ep[:] = to_np(env.t_ep)
    b.episode[:] = to_np(env.episode).view(np.uint32)
    t_g0 = env.t_g
    pw = W.policy_weights(w, 0.05)
    vw = W.value_weights(w)
    obs = torch.empty((T, 18, n), device="cuda")
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    grad = torch.empty(pw.size, device="cuda")
    coef = torch.full((T,), 1.0 / (n * T), device="cuda")
    env.shac_window(torch.from_numpy(pw).cuda(), torch.from_numpy(vw).cuda(), coef, 0.5 / n, grad,
                    obs=obs, rew=rew, done=done)
    m = oracle.model(w)
    ref = oracle.rollout(m, b, pw, None, t_g0, T, want=("obs", "rew"))
    assert np.abs(to_np(obs) - ref["obs"]).max() <= 1e-4
    assert np.array_equal(to_np(done), ref["done"])
    # critic values of every step and of the final observation, TD(lambda) targets
    val = torch.empty((T, n), device="cuda")
    env.value(obs, val)
    last_obs = torch.empty((1, 18, n), device="cuda")
    env.observe(last_obs[0])
    last = torch.empty((1, n), device="cuda")
    env.value(last_obs, last)
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    env.gae(rew, done, val, last[0], 0.99, 0.95, adv, ret)
    r_adv, r_ret = P.gae(to_np(rew), to_np(done), to_np(val), to_np(last[0]), 0.99, 0.95)
    assert np.abs(to_np(ret) - r_ret).max() <= 2e-5 * max(1.0, np.abs(r_ret).max())
    # critic regression on (obs, targets)
    L = auvenv.Learner(18, 8, H, 512, precision="fp32", seed=4, value_only=True, vf_coef=1.0)
    L.set_weights(pw, vw)
    g = torch.empty(L.n_policy + L.n_value, device="cuda")
    L.grads(dict(obs=obs, ret=ret), 0, 1, grad=g)
    host = dict(obs=to_np(obs), ret=to_np(ret), act=np.zeros((T, 8, n), np.float32),
                logp=np.zeros((T, n), np.float32), adv=np.zeros((T, n), np.float32))
    hp = dict(clip_eps=0.2, vf_coef=1.0, ent_coef=0.0, max_grad_norm=0.5, lr=3e-4,
              adam_beta1=0.9, adam_beta2=0.999, adam_eps=1e-8, logstd_min=-5.0,
              logstd_max=2.0, norm_adv=True, value_only=True)
    _, g_ref = P.Learner(pw, vw, (18, H, 8), hp, seed=4).grads(host, 0, 1, 512)
    gv, rv = to_np(g)[L.n_policy:], g_ref[L.n_policy:]
    assert np.abs(gv - rv).max() <= 1e-4 * np.abs(rv).max()


def test_shac_window_tf32(oracle):
    """The window with tensor-core (tf32) network products: J and the
    projected gradient against the oracle within tf32's tolerance (the
    operands carry 10 mantissa bits; measured values in the print)."""
    torch = need_gpu()
    n, T, H = 256, 8, 64
    w = W.workload("ppo_65536", n_envs=n, hidden=H, mlp="fp32", w_vs=0.05)
    env = make_env(w, policy=False)
    env.reset()
    pw = _smooth(W.policy_weights(w, 0.05), H)
    vw = W.value_weights(w, 0.1)
    b = oracle.Batch(np.arange(n))
    b.state[:] = to_np(env.state)
    b.params[:] = to_np(env.params)
    b.t_ep[:] = to_np(env.t_ep)
    b.episode[:] = to_np(env.episode).view(np.uint32)
    t_g0 = env.t_g
    coef = np.full(T, 1.0 / n, np.float32)
    grad = torch.empty(pw.size, device="cuda")
    J = torch.empty(n, device="cuda")
    env.shac_window(torch.from_numpy(pw).cuda(), torch.from_numpy(vw).cuda(),
                    torch.from_numpy(coef).cuda(), 0.5 / n, grad, J=J, precision="tf32")
    m = oracle.model(w)
    rng = np.random.default_rng(2)
    g = to_np(grad).astype(np.float64)
    worst = 0.0
    for _ in range(3):
        d = rng.normal(size=pw.size)
        Jr, dJ = oracle.shac_window(m, b, pw, d, vw, t_g0, T, coef, 0.5 / n)
        worst = max(worst, abs(g @ d - dJ.sum()) / np.abs(g * d).sum())
    jerr = np.abs(to_np(J) - Jr).max() / np.abs(Jr).max()
    print(f"[shac tf32] projected {worst:.3e}, J {jerr:.3e}")
    assert worst <= 5e-4 and jerr <= 5e-4        # measured 2.4e-5, 1.1e-5
