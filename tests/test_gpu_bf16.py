"""GPU parity of the tensor-core (tcgen05, bf16) network path against the
oracle's bf16 emulation (bf16 weights, inputs and hidden activations, exact
accumulation, fp32 biases, exact tanh).

Tolerances: the kernel adds the fp32 bias to the fp32 accumulator, applies
the hardware fp32 tanh (relative error about 2^-11) and rounds to bf16, so a
hidden unit is the oracle's correctly rounded value or a neighbour of it
when the exact value lies within 2^-11 of a rounding boundary; the inputs
of each layer are the same bf16 values up to those flips and the
accumulation order.  With N(0, 1/fan_in) weights these independent errors
add in quadrature through the 256-wide layers to about 2e-3 on outputs of
order one; BF16_HEAD_TOL (1e-2) bounds them with a margin of five.  Every
test reports the measured maximum next to it."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import STATE_TOL, assert_close, make_env, need_gpu, oracle_batch, to_np

pytestmark = pytest.mark.gpu

BF16_HEAD_TOL = 1e-2      # absolute, network outputs of order 1
BF16_VALUE_TOL = 1e-2


def _report(name, err, tol):
    print(f"[bf16 parity] {name}: max abs err {err:.3e} (tol {tol:.1e})")


@pytest.mark.parametrize("n", [1, 127, 1000, 40000])
def test_bf16_policy_and_value_forward(oracle, n):
    torch = need_gpu()
    w = W.workload("ppo_65536", n_envs=64)
    env = make_env(w, bias_std=0.1)
    obs = W.random_observations(3, n)
    head = torch.empty((n, 16), device="cuda")
    val = torch.empty((n,), device="cuda")
    env.policy_forward(torch.from_numpy(obs).cuda(), head, val)
    assert env.status().code == 0
    pw, vw = W.policy_weights(w, 0.1), W.value_weights(w, 0.1)
    idx = np.unique(np.r_[0, n - 1, np.random.default_rng(0).integers(0, n, 300)])
    ref_h = oracle.mlp(pw, 18, 256, 16, True, obs[idx].astype(np.float64))
    ref_v = oracle.mlp(vw, 18, 256, 1, True, obs[idx].astype(np.float64))[:, 0]
    eh = np.abs(to_np(head)[idx] - ref_h).max()
    ev = np.abs(to_np(val)[idx] - ref_v).max()
    _report(f"policy head n={n}", eh, BF16_HEAD_TOL)
    _report(f"value n={n}", ev, BF16_VALUE_TOL)
    assert eh <= BF16_HEAD_TOL and ev <= BF16_VALUE_TOL


def test_bf16_value_over_trajectory_layout(oracle):
    """env_value on obs[T][18][N] (the trajectory layout) with a ragged N."""
    torch = need_gpu()
    n, T = 1000, 7
    w = W.workload("ppo_65536", n_envs=n)
    env = make_env(w, bias_std=0.1)
    obs = W.random_observations(4, T * n).reshape(T, n, 18).transpose(0, 2, 1).copy()
    val = torch.empty((T, n), device="cuda")
    env.value(torch.from_numpy(obs).cuda(), val)
    vw = W.value_weights(w, 0.1)
    g = to_np(val)
    for t in (0, 3, 6):
        idx = np.r_[0, 1, 500, 999]
        ref = oracle.mlp(vw, 18, 256, 1, True, obs[t][:, idx].T.astype(np.float64))[:, 0]
        assert np.abs(g[t, idx] - ref).max() <= BF16_VALUE_TOL


@pytest.mark.parametrize("name", ["ppo_65536", "paper_4096"])
def test_bf16_value_many_tiles_per_group(oracle, name):
    """env_value over a trajectory of 3,909 row tiles: four groups per CTA,
    each serving 6 or 7 tiles in turn through the shared accumulators;
    ragged N (5,003) and both observation widths (18 and 12)."""
    torch = need_gpu()
    n, T = 5003, 100
    w = W.workload(name, n_envs=n)
    d = W.obs_dim(w)
    env = make_env(w, bias_std=0.1)
    obs = W.random_observations(5, T * n, d).reshape(T, n, d).transpose(0, 2, 1).copy()
    val = torch.full((T, n), float("nan"), device="cuda")
    env.value(torch.from_numpy(obs).cuda(), val)
    assert env.status().code == 0
    g = to_np(val)
    assert np.isfinite(g).all()
    vw = W.value_weights(w, 0.1)
    rng = np.random.default_rng(7)
    for t in (0, 1, 37, 98, 99):
        idx = np.unique(np.r_[0, 127, 128, n - 1, rng.integers(0, n, 60)])
        ref = oracle.mlp(vw, d, 256, 1, True, obs[t][:, idx].T.astype(np.float64))[:, 0]
        err = np.abs(g[t, idx] - ref).max()
        assert err <= BF16_VALUE_TOL, f"t={t}: {err:.3e}"


@pytest.mark.parametrize("n,T", [(65536, 128), (1048576, 4), (1000, 20), (300, 9)])
def test_bf16_rollout(oracle, n, T):
    """The rollout as the benchmark launches it (65,536 envs x 128 steps; the
    sweep's largest batch, 1,048,576 envs, several waves of CTAs; ragged
    small batches).  Step 0 starts from the
    bit-exact reset state: its observation is compared at the fp32 tolerance,
    its action, log-probability and value at the bf16 tolerance.  The episode
    length equals T, so every env ends its episode on the last step and the
    state buffers must hold the next episode's reset draw bit for bit.  Dones
    are bit-exact throughout."""
    torch = need_gpu()
    w = W.workload("ppo_65536", n_envs=n, episode_len=T)
    env = make_env(w)
    env.reset()
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    st = env.status()
    assert st.code == 0, (st.code, st.timeouts)
    g = {k: to_np(v) for k, v in traj.items()}
    assert np.all(np.isfinite(g["obs"])) and np.all(np.isfinite(g["rew"]))
    m = oracle.model(w)
    ids = np.unique(np.r_[0, n - 1, np.random.default_rng(5).integers(0, n, 12)])
    b = oracle_batch(oracle, m, ids)
    out = oracle.rollout(m, b, W.policy_weights(w), W.value_weights(w), 0, 1)
    assert_close(g["obs"][0][:, ids], out["obs"][0], STATE_TOL, what="obs[0]")
    ea = np.abs(g["act"][0][:, ids] - out["act"][0]).max()
    ev = np.abs(g["value"][0][ids] - out["value"][0]).max()
    el = np.abs(g["logp"][0][ids] - out["logp"][0]).max()
    _report(f"rollout n={n} act[0]", ea, BF16_HEAD_TOL * 8)
    _report(f"rollout n={n} value[0]", ev, BF16_VALUE_TOL)
    _report(f"rollout n={n} logp[0]", el, BF16_HEAD_TOL * 8)
    # a = mu + sigma eps with sigma = exp(log-std head), |eps| < 6
    assert ea <= BF16_HEAD_TOL * 8 and el <= BF16_HEAD_TOL * 8 and ev <= BF16_VALUE_TOL
    expect_done = np.zeros((T, n), np.uint8)
    expect_done[T - 1] = 1
    assert np.array_equal(g["done"], expect_done)
    fresh = oracle.Batch(np.arange(n))
    oracle.reset(m, fresh)
    oracle.reset(m, fresh)
    assert np.array_equal(to_np(env.state).view(np.uint32),
                          fresh.state.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.params).view(np.uint32),
                          fresh.params.astype(np.float32).view(np.uint32))


def test_bf16_rollout_is_deterministic(oracle):
    torch = need_gpu()
    w = W.workload("ppo_65536", n_envs=3000)
    e1, e2 = make_env(w), make_env(w)
    e1.reset()
    e2.reset()
    t1, t2 = e1.alloc_traj(10), e2.alloc_traj(10)
    e1.rollout(10, t1)
    e2.rollout(10, t2)
    for k in t1:
        assert torch.equal(t1[k], t2[k]), k
    assert torch.equal(e1.state, e2.state)


def test_sharded_batches_reproduce_the_full_batch(oracle):
    """Two shards with env_id_base = 0 and n reproduce one batch of 2n envs
    bit for bit (the multi-GPU partition, run here on one GPU)."""
    torch = need_gpu()
    n, T = 1000, 12
    full_w = W.workload("ppo_65536", n_envs=2 * n, episode_len=7)
    full = make_env(full_w)
    full.reset()
    tf = full.alloc_traj(T)
    full.rollout(T, tf)
    for r in range(2):
        w = dict(full_w, n_envs=n, env_id_base=r * n)
        e = make_env(w)
        e.reset()
        t = e.alloc_traj(T)
        e.rollout(T, t)
        sl = slice(r * n, (r + 1) * n)
        for k in ("obs", "act", "logp", "rew", "done", "value"):
            assert torch.equal(t[k], tf[k][..., sl]), k
        assert torch.equal(e.state, full.state[:, sl])
