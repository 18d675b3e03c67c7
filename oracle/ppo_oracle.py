"""TEST INFRASTRUCTURE: the oracle of the PPO learner's on-GPU pieces
(paper §III-A: PPO with its clipped surrogate objective, Schulman et al.
2017).  Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline /
reference legs may import this module; it shares nothing with the CUDA
library.  Plain numpy in float64.

Generalised advantage estimation (Schulman, Moritz, Levine, Jordan, Abbeel,
"High-dimensional continuous control using generalized advantage
estimation", ICLR 2016), over a trajectory in the rollout's layout
[T][N] (step t of env i at t*N + i):

  delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,   V_T = bootstrap value
  A_t     = delta_t + gamma lambda (1 - d_t) A_{t+1},  A_T = 0
  R_t     = A_t + V_t                              (the value target)

d_t = 1 marks the last step of an episode: nothing of the next episode (its
reset state's value, its rewards) flows back across it.

The minibatch update of PPO (clipped surrogate, value and entropy terms,
chain-rule gradients of the two tanh MLPs, global-norm clipping, Adam) and
the learner that runs epochs of minibatches drawn by the Feistel permutation
of the C++ oracle (oracle_minibatch_perm).  With hp["value_only"] the loss is
the value term alone (the critic regression of SHAC, whose targets are the
TD(lambda) returns = the GAE returns above) and the policy is not trained.  The paper names PPO but prints
none of its constants or loss weights: every hyperparameter is an input.
"""
from __future__ import annotations

import numpy as np


def gae(rew, done, value, last_value, gamma: float, lam: float):
    """Advantages and returns [T][N] (float64) by the backward recursion."""
    rew = np.asarray(rew, dtype=np.float64)
    value = np.asarray(value, dtype=np.float64)
    nonterm = 1.0 - np.asarray(done, dtype=np.float64)
    T, n = rew.shape
    adv = np.zeros((T, n))
    a_next = np.zeros(n)
    v_next = np.asarray(last_value, dtype=np.float64)
    for t in range(T - 1, -1, -1):
        delta = rew[t] + gamma * nonterm[t] * v_next - value[t]
        a_next = delta + gamma * lam * nonterm[t] * a_next
        adv[t] = a_next
        v_next = value[t]
    return adv, adv + value


# ---------------------------------------------------------------------------
# PPO minibatch update (Schulman et al. 2017, the clipped surrogate objective
# the paper names in §III-A), float64, in plain steps:
#   forward  h1 = tanh(W1 x + b1), h2 = tanh(W2 h1 + b2), y = W3 h2 + b3
#   policy   mu = y[:A], ls = clip(y[A:2A], lo, hi), sigma = exp(ls)
#            logp = sum_k -((a - mu)/sigma)^2 / 2 - ls - log(2 pi) / 2
#            r = exp(logp - logp_old)
#            A_n = (A - mean A) / (std A + 1e-8)      (per minibatch, ddof 1)
#   loss     L = mean(max(-A_n r, -A_n clip(r, 1 - eps, 1 + eps)))
#              + c_v mean((V - R)^2) / 2 - c_ent mean(sum_k ls_k + (1 + log 2 pi) / 2)
#   backward by the chain rule (no gradient where the log-std clamp is active)
#   Adam     m = b1 m + (1 - b1) g, v = b2 v + (1 - b2) g^2,
#            w -= lr (m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) + eps_adam)
# Weights are the flat [W1 | b1 | W2 | b2 | W3 | b3] arrays of the rollout.
# ---------------------------------------------------------------------------
LOG_2PI = float(np.log(2.0 * np.pi))


def gaussian_policy(y, a, hp):
    """Policy head y [B][2A] -> mean, clamped log-std, mask of samples whose
    log-std lies inside the clamp, and the diagonal-Gaussian log-density of
    the actions a [B][A]."""
    A = a.shape[1]
    mu, raw = y[:, :A], y[:, A:2 * A]
    ls = np.clip(raw, hp["logstd_min"], hp["logstd_max"])
    inside = (raw >= hp["logstd_min"]) & (raw <= hp["logstd_max"])
    z = (a - mu) / np.exp(ls)
    logp = np.sum(-0.5 * z * z - ls - 0.5 * LOG_2PI, axis=1)
    return mu, ls, inside, logp


def unpack(w, in_dim, H, out):
    w = np.asarray(w, dtype=np.float64)
    sizes = [H * in_dim, H, H * H, H, out * H, out]
    parts, o = [], 0
    for s in sizes:
        parts.append(w[o:o + s])
        o += s
    W1, b1, W2, b2, W3, b3 = parts
    return W1.reshape(H, in_dim), b1, W2.reshape(H, H), b2, W3.reshape(out, H), b3


def mlp_forward(w, in_dim, H, out, x):
    """x [B][in_dim] -> (h1 [B][H], h2 [B][H], y [B][out])."""
    W1, b1, W2, b2, W3, b3 = unpack(w, in_dim, H, out)
    h1 = np.tanh(x @ W1.T + b1)
    h2 = np.tanh(h1 @ W2.T + b2)
    return h1, h2, h2 @ W3.T + b3


def mlp_backward(w, in_dim, H, out, x, h1, h2, g_y):
    """Gradient of sum(g_y * y) with respect to the flat weights."""
    W1, b1, W2, b2, W3, b3 = unpack(w, in_dim, H, out)
    gW3 = g_y.T @ h2
    gb3 = g_y.sum(axis=0)
    g_z2 = (g_y @ W3) * (1.0 - h2 * h2)
    gW2 = g_z2.T @ h1
    gb2 = g_z2.sum(axis=0)
    g_z1 = (g_z2 @ W2) * (1.0 - h1 * h1)
    gW1 = g_z1.T @ x
    gb1 = g_z1.sum(axis=0)
    return np.concatenate([gW1.ravel(), gb1, gW2.ravel(), gb2, gW3.ravel(), gb3])


def ppo_loss(pw, vw, dims, x, a, logp_old, adv, ret, hp):
    """Scalar loss and its parts (forward only; used by the pins)."""
    in_dim, H, A = dims
    _, _, y = mlp_forward(pw, in_dim, H, 2 * A, x)
    _, _, v = mlp_forward(vw, in_dim, H, 1, x)
    _, ls, _, logp = gaussian_policy(y, a, hp)
    r = np.exp(logp - logp_old)
    an = (adv - adv.mean()) / (adv.std(ddof=1) + 1e-8) if hp["norm_adv"] else adv
    eps = hp["clip_eps"]
    pg = np.mean(np.maximum(-an * r, -an * np.clip(r, 1 - eps, 1 + eps)))
    vl = 0.5 * np.mean((v[:, 0] - ret) ** 2)
    ent = np.mean(np.sum(ls + 0.5 * (1.0 + LOG_2PI), axis=1))
    kl = float(np.mean(logp_old - logp))
    cf = float(np.mean(np.abs(r - 1.0) > eps))
    if hp.get("value_only"):
        # critic regression (SHAC's value step): only the value term
        pg, ent, kl, cf = 0.0, 0.0, 0.0, 0.0
        return hp["vf_coef"] * vl, dict(pg_loss=pg, v_loss=vl, entropy=ent, approx_kl=kl,
                                        clip_frac=cf)
    loss = pg + hp["vf_coef"] * vl - hp["ent_coef"] * ent
    return loss, dict(pg_loss=pg, v_loss=vl, entropy=ent, approx_kl=kl, clip_frac=cf)


def ppo_grads(pw, vw, dims, x, a, logp_old, adv, ret, hp):
    """(loss parts, policy gradient, value gradient) by the chain rule."""
    in_dim, H, A = dims
    B = x.shape[0]
    h1, h2, y = mlp_forward(pw, in_dim, H, 2 * A, x)
    vh1, vh2, v = mlp_forward(vw, in_dim, H, 1, x)
    mu, ls, inside, logp = gaussian_policy(y, a, hp)
    sig2 = np.exp(2.0 * ls)
    d = a - mu
    r = np.exp(logp - logp_old)
    an = (adv - adv.mean()) / (adv.std(ddof=1) + 1e-8) if hp["norm_adv"] else adv
    eps = hp["clip_eps"]
    unclipped = np.where(an > 0, r <= 1 + eps, r >= 1 - eps)
    g_logp = np.where(unclipped, -an * r, 0.0) / B
    g_y = np.zeros_like(y)
    g_y[:, :A] = g_logp[:, None] * d / sig2
    g_y[:, A:] = (g_logp[:, None] * (d * d / sig2 - 1.0) - hp["ent_coef"] / B) * inside
    g_v = hp["vf_coef"] * (v - ret[:, None]) / B
    if hp.get("value_only"):
        g_y = np.zeros_like(g_y)
    gp = mlp_backward(pw, in_dim, H, 2 * A, x, h1, h2, g_y)
    gv = mlp_backward(vw, in_dim, H, 1, x, vh1, vh2, g_v)
    _, parts = ppo_loss(pw, vw, dims, x, a, logp_old, adv, ret, hp)
    return parts, gp, gv


def adam(w, g, m, v, t, hp):
    """One Adam step (t counts from 1); returns new (w, m, v)."""
    b1, b2 = hp["adam_beta1"], hp["adam_beta2"]
    m = b1 * m + (1 - b1) * g
    v = b2 * v + (1 - b2) * g * g
    mh = m / (1 - b1 ** t)
    vh = v / (1 - b2 ** t)
    return w - hp["lr"] * mh / (np.sqrt(vh) + hp["adam_eps"]), m, v


def gather_minibatch(obs, act, logp, adv, ret, idx):
    """Rows r = t*N + i of trajectory arrays obs[T][D][N], act[T][A][N] and
    [T][N] arrays -> x [B][D], a [B][A], logp, adv, ret [B]."""
    T, D, N = obs.shape
    t, i = np.asarray(idx) // N, np.asarray(idx) % N
    return (obs[t, :, i].astype(np.float64), act[t, :, i].astype(np.float64),
            logp[t, i].astype(np.float64), adv[t, i].astype(np.float64),
            ret[t, i].astype(np.float64))


def clip_by_global_norm(g, max_norm: float):
    """Scale g so that its 2-norm is at most max_norm (no clipping when
    max_norm <= 0); the scale is max_norm / (norm + 1e-6), capped at 1.
    Returns (scaled g, norm before clipping)."""
    norm = float(np.sqrt(np.sum(np.asarray(g, dtype=np.float64) ** 2)))
    if max_norm <= 0:
        return g, norm
    return g * min(1.0, max_norm / (norm + 1e-6)), norm


class Learner:
    """Weights, Adam moments and counters of one PPO learner.  The two
    networks' parameters form one vector [policy | value] for the gradient
    norm and for Adam."""

    def __init__(self, pw, vw, dims, hp, seed: int):
        self.dims = tuple(dims)
        self.hp = dict(hp)
        self.seed = int(seed)
        self.n_policy = len(pw)
        self.w = np.concatenate([np.asarray(pw, np.float64), np.asarray(vw, np.float64)])
        self.m = np.zeros_like(self.w)
        self.v = np.zeros_like(self.w)
        self.t = 0          # Adam steps taken
        self.epoch = 0      # next global epoch number

    @property
    def policy(self):
        return self.w[:self.n_policy]

    @property
    def value(self):
        return self.w[self.n_policy:]

    def minibatch(self, traj, epoch: int, j: int, B: int):
        """Samples at positions j*B .. j*B+B-1 of the epoch's permutation of
        the T*N trajectory rows (row r = t*N + i)."""
        from oracle import oracle as O
        T, _, N = traj["obs"].shape
        idx = O.minibatch_perm(self.seed, epoch, T * N, j * B, B).astype(np.int64)
        return gather_minibatch(traj["obs"], traj["act"], traj["logp"], traj["adv"],
                                traj["ret"], idx)

    def grads(self, traj, epoch: int, j: int, B: int):
        x, a, lp, ad, rt = self.minibatch(traj, epoch, j, B)
        parts, gp, gv = ppo_grads(self.policy, self.value, self.dims, x, a, lp, ad, rt, self.hp)
        return parts, np.concatenate([gp, gv])

    def apply(self, g):
        g, norm = clip_by_global_norm(g, self.hp["max_grad_norm"])
        self.t += 1
        self.w, self.m, self.v = adam(self.w, g, self.m, self.v, self.t, self.hp)
        return norm

    def update(self, traj, epochs: int, n_minibatches: int, B: int):
        """epochs x n_minibatches gradient steps; returns the mean over the
        steps of the loss parts and of the gradient norm before clipping."""
        T, _, N = traj["obs"].shape
        assert n_minibatches * B <= T * N
        acc = {}
        for _ in range(epochs):
            for j in range(n_minibatches):
                parts, g = self.grads(traj, self.epoch, j, B)
                parts = dict(parts, grad_norm=self.apply(g))
                for k, val in parts.items():
                    acc[k] = acc.get(k, 0.0) + float(val)
            self.epoch += 1
        return {k: val / (epochs * n_minibatches) for k, val in acc.items()}
