"""Pins for the PPO learner's oracle.

Generalised advantage estimation against formulations that do not share its
recursion: the lambda = 1 case is the discounted Monte-Carlo return minus
the value (summed explicitly per episode), lambda = 0 is the one-step TD
error, the general case equals the lambda-weighted sum of n-step advantages
(the definition GAE is derived from), and a 3-step example computed by hand.

The minibatch update: the Gaussian log-density and entropy against scipy,
the hand-written gradients against central differences and torch autograd,
hand-computed clipped-surrogate cases, the first-epoch and value-loss
special cases, Adam and global-norm clipping against torch.optim.Adam and
clip_grad_norm_, the Feistel minibatch permutation (bijection, inverse,
keyed, even spread), the gather's row mapping, and the learner's counters."""
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


# ---------------------------------------------------------------------------
# PPO minibatch update: loss, gradients, clipping, Adam, permutation.
# ---------------------------------------------------------------------------
HP = dict(clip_eps=0.2, vf_coef=0.5, ent_coef=0.01, max_grad_norm=0.5, lr=3e-4,
          adam_beta1=0.9, adam_beta2=0.999, adam_eps=1e-8, logstd_min=-5.0, logstd_max=2.0,
          norm_adv=True)


def _net(rng, in_dim, H, out, scale=0.6):
    n = H * in_dim + H + H * H + H + out * H + out
    return rng.normal(size=n) * scale


def _problem(seed, in_dim=5, H=7, A=3, B=24, ratio_spread=0.4):
    """Random small networks and a minibatch whose old log-probs put ratios
    on both sides of the clip range."""
    rng = np.random.default_rng(seed)
    pw, vw = _net(rng, in_dim, H, 2 * A), _net(rng, in_dim, H, 1)
    x = rng.normal(size=(B, in_dim))
    _, _, y = P.mlp_forward(pw, in_dim, H, 2 * A, x)
    a = y[:, :A] + rng.normal(size=(B, A)) * np.exp(np.clip(y[:, A:], -5, 2))
    _, _, _, lp = P.gaussian_policy(y, a, HP)
    lp_old = lp + rng.normal(size=B) * ratio_spread
    adv = rng.normal(size=B)
    ret = rng.normal(size=B)
    return pw, vw, (in_dim, H, A), x, a, lp_old, adv, ret


def test_gaussian_logp_and_entropy_match_scipy():
    stats = pytest.importorskip("scipy.stats")
    rng = np.random.default_rng(5)
    y = rng.normal(size=(6, 8)) * 2.0          # some log-stds beyond the clamp
    a = rng.normal(size=(6, 4))
    mu, ls, inside, logp = P.gaussian_policy(y, a, HP)
    for b in range(6):
        sd = np.exp(np.clip(y[b, 4:], -5.0, 2.0))
        assert logp[b] == pytest.approx(stats.norm.logpdf(a[b], y[b, :4], sd).sum(), rel=1e-12)
        ent = stats.multivariate_normal(mean=np.zeros(4), cov=np.diag(sd ** 2)).entropy()
        assert np.sum(ls[b] + 0.5 * (1 + P.LOG_2PI)) == pytest.approx(ent, rel=1e-12)
    assert np.array_equal(inside, (y[:, 4:] >= -5) & (y[:, 4:] <= 2))


def test_loss_gradients_match_finite_differences():
    """Central differences of the scalar loss in every 7th parameter of both
    networks, with ratios inside and outside the clip range and log-stds
    inside the clamp (the loss is smooth there)."""
    pw, vw, dims, x, a, lp_old, adv, ret = _problem(11)
    _, gp, gv = P.ppo_grads(pw, vw, dims, x, a, lp_old, adv, ret, HP)
    h = 1e-6
    for w, g, which in ((pw, gp, 0), (vw, gv, 1)):
        for k in range(0, len(w), 7):
            wp, wm = w.copy(), w.copy()
            wp[k] += h
            wm[k] -= h
            args = (wp, vw) if which == 0 else (pw, wp)
            lp_ = P.ppo_loss(*args, dims, x, a, lp_old, adv, ret, HP)[0]
            args = (wm, vw) if which == 0 else (pw, wm)
            lm_ = P.ppo_loss(*args, dims, x, a, lp_old, adv, ret, HP)[0]
            assert g[k] == pytest.approx((lp_ - lm_) / (2 * h), rel=1e-5, abs=1e-8), (which, k)


def test_loss_gradients_match_torch_autograd():
    """The same loss built from torch float64 ops, differentiated by autograd:
    pins the hand-written chain rule of every layer, the clamp mask and the
    clip branches."""
    torch = pytest.importorskip("torch")
    pw, vw, dims, x, a, lp_old, adv, ret = _problem(12, ratio_spread=1.0)
    in_dim, H, A = dims
    parts, gp, gv = P.ppo_grads(pw, vw, dims, x, a, lp_old, adv, ret, HP)
    T = lambda v: torch.tensor(v, dtype=torch.float64)
    tp, tv = T(pw).requires_grad_(), T(vw).requires_grad_()

    def net(w, out):
        o = 0
        mats = []
        for r, c in ((H, in_dim), (H, H), (out, H)):
            Wm = w[o:o + r * c].reshape(r, c)
            o += r * c
            bv = w[o:o + r]
            o += r
            mats.append((Wm, bv))
        h = torch.tanh(T(x) @ mats[0][0].T + mats[0][1])
        h = torch.tanh(h @ mats[1][0].T + mats[1][1])
        return h @ mats[2][0].T + mats[2][1]

    y, v = net(tp, 2 * A), net(tv, 1)[:, 0]
    dist = torch.distributions.Normal(y[:, :A], torch.exp(torch.clamp(y[:, A:], -5.0, 2.0)))
    logp = dist.log_prob(T(a)).sum(1)
    r = torch.exp(logp - T(lp_old))
    an = (T(adv) - T(adv).mean()) / (T(adv).std() + 1e-8)
    pg = torch.max(-an * r, -an * torch.clamp(r, 0.8, 1.2)).mean()
    loss = pg + 0.5 * 0.5 * ((v - T(ret)) ** 2).mean() - 0.01 * dist.entropy().sum(1).mean()
    loss.backward()
    loss = loss.detach()
    assert loss.item() == pytest.approx(P.ppo_loss(pw, vw, dims, x, a, lp_old, adv, ret, HP)[0],
                                        rel=1e-12)
    assert np.allclose(tp.grad.numpy(), gp, rtol=1e-10, atol=1e-13)
    assert np.allclose(tv.grad.numpy(), gv, rtol=1e-10, atol=1e-13)
    assert 0.0 < parts["clip_frac"] < 1.0


def test_surrogate_hand_cases():
    """Two samples, unnormalised advantages, ratios fixed through the old
    log-probs: r = 1.5 with A = +2 is clipped to 1.2 (term -2.4); r = 1.5
    with A = -1 keeps the unclipped, pessimistic value (term +1.5)."""
    pw, vw, dims, x, a, _, _, _ = _problem(13, B=2)
    hp = dict(HP, norm_adv=False, vf_coef=0.0, ent_coef=0.0)
    in_dim, H, A = dims
    _, _, y = P.mlp_forward(pw, in_dim, H, 2 * A, x)
    _, _, _, lp = P.gaussian_policy(y, a, hp)
    lp_old = lp - np.log(1.5)
    loss, parts = P.ppo_loss(pw, vw, dims, x, a, lp_old, np.array([2.0, -1.0]), np.zeros(2), hp)
    assert parts["pg_loss"] == pytest.approx((-2.4 + 1.5) / 2, rel=1e-12)
    assert loss == pytest.approx(parts["pg_loss"], rel=1e-15)
    assert parts["clip_frac"] == 1.0
    assert parts["approx_kl"] == pytest.approx(-np.log(1.5), rel=1e-12)
    # the clipped sample has no policy gradient: only sample 1 contributes
    _, g_both, _ = P.ppo_grads(pw, vw, dims, x, a, lp_old, np.array([2.0, -1.0]), np.zeros(2), hp)
    _, g_one, _ = P.ppo_grads(pw, vw, dims, x, a, lp_old, np.array([0.0, -1.0]), np.zeros(2), hp)
    assert np.allclose(g_both, g_one, rtol=1e-13, atol=1e-16)


def test_first_epoch_surrogate_and_value_loss():
    """At the rollout policy (r = 1) the normalised surrogate is -mean(A_n) =
    0; the value loss is 0 at R = V and 1/2 at R = V - 1."""
    pw, vw, dims, x, a, _, adv, _ = _problem(14)
    in_dim, H, A = dims
    _, _, y = P.mlp_forward(pw, in_dim, H, 2 * A, x)
    _, _, _, lp = P.gaussian_policy(y, a, HP)
    _, _, v = P.mlp_forward(vw, in_dim, H, 1, x)
    _, parts = P.ppo_loss(pw, vw, dims, x, a, lp, adv, v[:, 0], HP)
    assert abs(parts["pg_loss"]) < 1e-15 and parts["v_loss"] == 0.0
    assert parts["approx_kl"] == 0.0 and parts["clip_frac"] == 0.0
    _, parts = P.ppo_loss(pw, vw, dims, x, a, lp, adv, v[:, 0] - 1.0, HP)
    assert parts["v_loss"] == pytest.approx(0.5, rel=1e-14)


def test_adam_and_clipping_match_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(15)
    hp = dict(HP, lr=1e-2)
    w = rng.normal(size=50)
    tw = torch.tensor(w, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.Adam([tw], lr=hp["lr"], betas=(hp["adam_beta1"], hp["adam_beta2"]),
                           eps=hp["adam_eps"])
    m, v = np.zeros(50), np.zeros(50)
    for t in range(1, 8):
        g = rng.normal(size=50) * (3.0 if t % 2 else 0.01)
        gc, norm = P.clip_by_global_norm(g, 0.5)
        tw.grad = torch.tensor(g, dtype=torch.float64)
        tnorm = torch.nn.utils.clip_grad_norm_([tw], 0.5)
        assert norm == pytest.approx(float(tnorm), rel=1e-14)
        assert np.allclose(tw.grad.numpy(), gc, rtol=1e-14, atol=0)
        opt.step()
        w, m, v = P.adam(w, gc, m, v, t, hp)
        assert np.allclose(tw.detach().numpy(), w, rtol=1e-13, atol=1e-15)
    g = rng.normal(size=5)
    assert P.clip_by_global_norm(g, 0.0)[0] is g


def test_minibatch_permutation_is_a_keyed_bijection():
    from oracle import oracle as O
    for m in (1, 2, 3, 4, 5, 16, 17, 1000, 4096, 4097, 70001):
        p = O.minibatch_perm(9, 2, m, 0, m)
        assert np.array_equal(np.sort(p), np.arange(m)), m
    # a Feistel pass is invertible; different epochs and seeds permute differently
    for x in (0, 1, 77, 1023):
        assert O.feistel(O.feistel(x, 1000, 5, 6), 1000, 5, 6, inverse=True) == x
    a = O.minibatch_perm(9, 2, 4096, 0, 4096)
    assert not np.array_equal(a, O.minibatch_perm(9, 3, 4096, 0, 4096))
    assert not np.array_equal(a, O.minibatch_perm(10, 2, 4096, 0, 4096))
    assert np.array_equal(a[100:300], O.minibatch_perm(9, 2, 4096, 100, 200))
    # positions spread evenly: over 400 epochs, where position 0 of [0, 8) lands
    hits = np.bincount([O.minibatch_perm(1, e, 8, 0, 1)[0] for e in range(400)], minlength=8)
    assert hits.min() > 25 and hits.max() < 80


def test_gather_minibatch_layout():
    T, D, N, A = 3, 4, 5, 2
    t, k, i = np.meshgrid(np.arange(T), np.arange(D), np.arange(N), indexing="ij")
    obs = (100 * t + 10 * k + i).astype(np.float32)
    t2, k2, i2 = np.meshgrid(np.arange(T), np.arange(A), np.arange(N), indexing="ij")
    act = (100 * t2 + 10 * k2 + i2).astype(np.float32)
    flat = (np.arange(T)[:, None] * 1000 + np.arange(N)[None]).astype(np.float32)
    x, a, lp, ad, rt = P.gather_minibatch(obs, act, flat, flat + 1, flat + 2, [0, 7, 14])
    assert np.array_equal(x[1], [100 + 2, 112, 122, 132])     # row 7: t = 1, i = 2
    assert np.array_equal(a[2], [200 + 4, 214])                # row 14: t = 2, i = 4
    assert np.array_equal(lp, [0, 1002, 2004]) and np.array_equal(rt, [2, 1004, 2006])


def test_learner_update_counts_and_moves():
    """Two epochs of three minibatches take six Adam steps and change both
    networks; with lr = 0 nothing moves."""
    rng = np.random.default_rng(16)
    in_dim, H, A, T, N = 4, 6, 2, 5, 40
    traj = dict(obs=rng.normal(size=(T, in_dim, N)), act=rng.normal(size=(T, A, N)),
                logp=rng.normal(size=(T, N)) - 3, adv=rng.normal(size=(T, N)),
                ret=rng.normal(size=(T, N)))
    pw, vw = _net(rng, in_dim, H, 2 * A), _net(rng, in_dim, H, 1)
    L = P.Learner(pw, vw, (in_dim, H, A), HP, seed=3)
    stats = L.update(traj, 2, 3, 64)
    assert L.t == 6 and L.epoch == 2
    assert not np.allclose(L.policy, pw) and not np.allclose(L.value, vw)
    assert set(stats) >= {"pg_loss", "v_loss", "entropy", "approx_kl", "clip_frac", "grad_norm"}
    L0 = P.Learner(pw, vw, (in_dim, H, A), dict(HP, lr=0.0), seed=3)
    L0.update(traj, 1, 2, 64)
    assert np.array_equal(L0.policy, pw) and np.array_equal(L0.value, vw)


def test_value_only_is_the_critic_regression():
    """value_only: the loss is c_v mean((V - R)^2) / 2, the policy gradient
    is zero, and the value gradient equals the full loss's (whose value part
    does not depend on the policy)."""
    pw, vw, dims, x, a, lp_old, adv, ret = _problem(17)
    hp = dict(HP, value_only=True)
    loss, parts = P.ppo_loss(pw, vw, dims, x, a, lp_old, adv, ret, hp)
    assert loss == pytest.approx(HP["vf_coef"] * parts["v_loss"], rel=1e-15)
    assert parts["pg_loss"] == 0.0 and parts["entropy"] == 0.0
    _, gp, gv = P.ppo_grads(pw, vw, dims, x, a, lp_old, adv, ret, hp)
    _, _, gv_full = P.ppo_grads(pw, vw, dims, x, a, lp_old, adv, ret, HP)
    assert np.all(gp == 0.0) and np.array_equal(gv, gv_full)
