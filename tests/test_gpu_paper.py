"""GPU parity of the paper's own environment (wrench action of Eq. 1,
inertia-box fluid model, effective gravity, 12-float axis-angle observation,
five-term reward of Eqs. 2-7) through the C ABI against the oracle's paper
model: resets bit-exact (including the zeroed action history), observation,
action replay and the fp32 closed-loop rollout within the fp32 tolerances of
the Fossen model, auto-resets inside the horizon, host trajectories equal to
device ones, and the tensor-core (bf16) networks and rollout within the bf16
tolerances of the Fossen model's tensor-core path."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import STATE_TOL, assert_close, make_env, need_gpu, to_np, u32

pytestmark = pytest.mark.gpu


def _oracle_batch(oracle, m, n, resets=1):
    b = oracle.PaperBatch(np.arange(n))
    for _ in range(resets):
        oracle.paper_reset(m, b)
    return b


@pytest.mark.parametrize("n,dr", [(64, 0), (999, 1), (4096, 1)])
def test_paper_reset_bit_exact(oracle, n, dr):
    torch = need_gpu()
    w = W.workload("paper_tiny", n_envs=n, dr_enable=dr, init_pos_range=0.4, init_att_range=0.3)
    env = make_env(w, policy=False)
    env.state.fill_(7.0)              # the reset must clear velocities and history
    env.reset()
    env.reset()
    m = oracle.paper_model(w)
    b = _oracle_batch(oracle, m, n, resets=2)
    assert np.array_equal(to_np(env.state).view(np.uint32),
                          b.state.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.params).view(np.uint32),
                          b.params.astype(np.float32).view(np.uint32))
    assert np.all(to_np(env.t_ep) == 0) and np.all(u32(env.episode) == 2)


def test_paper_observation(oracle):
    torch = need_gpu()
    n = 777
    w = W.workload("paper_tiny", n_envs=n, dr_enable=1)
    env = make_env(w, policy=False)
    env.reset()
    rng = np.random.default_rng(4)
    st = to_np(env.state).copy()
    q = rng.standard_normal((4, n))
    st[3:7] = q / np.linalg.norm(q, axis=0)
    st[0:3] = rng.uniform(-2, 2, (3, n))
    st[7:13] = rng.uniform(-1, 1, (6, n))
    env.state.copy_(torch.from_numpy(st))
    obs = torch.empty((12, n), device="cuda")
    env.observe(obs)
    got = to_np(obs)
    pr = to_np(env.params)
    for i in list(range(0, n, 37)) + [n - 1]:
        ref = oracle.paper_observe(st[:, i].astype(np.float64), pr[:, i].astype(np.float64))
        assert_close(got[:, i], ref, 1e-5, what=f"obs env {i}")


@pytest.mark.parametrize("n,T,L,K", [(999, 60, 23, 4), (4096, 40, 500, 8), (64, 30, 7, 1)])
def test_paper_replay_against_oracle(oracle, n, T, L, K):
    """Per-step state (trace, history rows included), reward and done over
    auto-resets; dones bit-exact."""
    torch = need_gpu()
    w = W.workload("paper_tiny", n_envs=n, substeps=4, dr_enable=1, episode_len=L, mavg_len=K,
                   g_eff=0.05, fluid_viscosity=0.01)
    env = make_env(w, policy=False)
    env.reset()
    m = oracle.paper_model(w)
    b = _oracle_batch(oracle, m, n)
    acts = W.replay_actions(3, T, n, scale=0.8, act=6)
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    trace = torch.empty((T, W.PAPER_STATE_FIELDS, n), device="cuda")
    env.step_actions(torch.from_numpy(acts).cuda(), rew, done, trace)
    r_rew, r_done, r_tr = oracle.paper_replay(m, b, acts, trace=True)
    assert np.array_equal(to_np(done), r_done)
    assert_close(to_np(rew), r_rew, STATE_TOL * 10, what="reward")
    assert_close(to_np(trace), r_tr, STATE_TOL, what="state trace")
    assert_close(to_np(env.state), b.state, STATE_TOL, what="final state")
    assert np.array_equal(to_np(env.t_ep), b.t_ep)
    assert np.array_equal(u32(env.episode), b.episode)


def test_paper_replay_full_episode_sampled(oracle):
    """The physics-only launch the benchmark times on the paper workload:
    4,096 envs x 512 steps (one whole episode, K = 4, gravity randomised),
    40 sampled envs against the oracle step by step (trace with history
    rows, reward); dones bit-exact, the last step's state the next reset."""
    torch = need_gpu()
    w = W.workload("paper_4096")
    n, T = int(w["n_envs"]), int(w["steps"])
    env = make_env(w, policy=False)
    env.reset()
    m = oracle.paper_model(w)
    ids = np.unique(np.r_[0, n - 1, np.random.default_rng(11).integers(0, n, 38)])
    b = oracle.PaperBatch(ids)
    oracle.paper_reset(m, b)
    acts = W.replay_actions(3, T, n, scale=0.8, act=6)
    rew = torch.empty((T, n), device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    trace = torch.empty((T, W.PAPER_STATE_FIELDS, n), device="cuda")
    env.step_actions(torch.from_numpy(acts).cuda(), rew, done, trace)
    assert env.status().code == 0
    r_rew, r_done, r_tr = oracle.paper_replay(m, b, np.ascontiguousarray(acts[:, :, ids]),
                                              trace=True)
    g_done = to_np(done)[:, ids]
    assert np.array_equal(g_done, r_done) and np.all(g_done[-1] == 1) and g_done[:-1].sum() == 0
    assert_close(to_np(rew)[:, ids], r_rew, STATE_TOL * 10, what="reward")
    assert_close(to_np(trace)[:, :, ids], r_tr, STATE_TOL, what="state trace")
    assert_close(to_np(env.state)[:, ids], b.state, STATE_TOL, what="final state")


@pytest.mark.parametrize("hidden,policy_out,has_value", [(64, 6, 0), (256, 12, 1)])
def test_paper_fp32_rollout_against_oracle(oracle, hidden, policy_out, has_value):
    torch = need_gpu()
    n, T = 500, 40
    w = W.workload("paper_tiny", n_envs=n, hidden=hidden, policy_out=policy_out,
                   has_value=has_value, substeps=4, episode_len=17, dr_enable=1)
    env = make_env(w)
    env.reset()
    keys = ("obs", "act", "logp", "rew", "done") + (("value",) if has_value else ())
    traj = env.alloc_traj(T, keys=keys)
    env.rollout(T, traj)
    m = oracle.paper_model(w)
    b = _oracle_batch(oracle, m, n)
    ref = oracle.paper_rollout(m, b, W.policy_weights(w),
                               W.value_weights(w) if has_value else None, 0, T)
    assert np.array_equal(to_np(traj["done"]), ref["done"])
    for k in ("obs", "act", "logp", "rew") + (("value",) if has_value else ()):
        assert_close(to_np(traj[k]), ref[k], 1e-4, what=k)
    assert_close(to_np(env.state), b.state, 1e-4, what="final state")


def test_paper_host_trajectory_matches_device():
    """The staged host path with the paper model's 12- and 6-row arrays."""
    torch = need_gpu()
    n, T = 3000, 21
    w = W.workload("paper_tiny", n_envs=n, has_value=1, episode_len=9)
    outs = []
    for host in (False, True):
        env = make_env(w)
        env.reset()
        traj = env.alloc_traj(T, pinned_host=host)
        env.rollout(T, traj)
        torch.cuda.synchronize()
        outs.append({k: to_np(v).copy() for k, v in traj.items()})
    for k in outs[0]:
        assert np.array_equal(outs[0][k], outs[1][k]), k


BF16_TOL = 1e-2     # network outputs, as for the Fossen model's bf16 path


@pytest.mark.parametrize("n", [1, 300, 40000])
def test_paper_bf16_forward(oracle, n):
    torch = need_gpu()
    w = W.workload("paper_4096", n_envs=64)
    env = make_env(w, bias_std=0.1)
    obs = W.random_observations(5, n, dim=12)
    head = torch.empty((n, 12), device="cuda")
    val = torch.empty((n,), device="cuda")
    env.policy_forward(torch.from_numpy(obs).cuda(), head, val)
    assert env.status().code == 0
    idx = np.unique(np.r_[0, n - 1, np.random.default_rng(0).integers(0, n, 200)])
    ref_h = oracle.mlp(W.policy_weights(w, 0.1), 12, 256, 12, True, obs[idx].astype(np.float64))
    ref_v = oracle.mlp(W.value_weights(w, 0.1), 12, 256, 1, True, obs[idx].astype(np.float64))
    eh = np.abs(to_np(head)[idx] - ref_h).max()
    ev = np.abs(to_np(val)[idx] - ref_v[:, 0]).max()
    print(f"[paper bf16] n={n}: head {eh:.3e} value {ev:.3e} (tol {BF16_TOL})")
    assert eh <= BF16_TOL and ev <= BF16_TOL


@pytest.mark.parametrize("T", [48, 512])
def test_paper_bf16_rollout(oracle, T):
    """The paper workload's tensor-core rollout over one whole episode
    (T = episode_len; 512 is the paper's episode and the benchmark's launch
    of 4,096 envs x 512 steps): step-0 observations to 1e-5, actions and
    log-probs within the bf16 head tolerance, dones exact, values against
    the oracle's bf16 value network, and the final state equal bit for bit
    to the next episode's reset draw (history cleared)."""
    torch = need_gpu()
    n = 4096
    w = W.workload("paper_4096", n_envs=n, episode_len=T)
    env = make_env(w)
    env.reset()
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    assert env.status().code == 0
    m = oracle.paper_model(w)
    sample = np.r_[0, 1, 2, 1000, 2047, 4095]
    b = oracle.PaperBatch(sample)
    oracle.paper_reset(m, b)
    ref = oracle.paper_rollout(m, b, W.policy_weights(w), W.value_weights(w), 0, 1)
    assert_close(to_np(traj["obs"])[0][:, sample], ref["obs"][0], 1e-5, what="obs step 0")
    assert np.abs(to_np(traj["act"])[0][:, sample] - ref["act"][0]).max() <= 0.24
    assert np.abs(to_np(traj["logp"])[0][sample] - ref["logp"][0]).max() <= 0.24
    assert np.abs(to_np(traj["value"])[0][sample] - ref["value"][0]).max() <= BF16_TOL
    done = to_np(traj["done"])
    assert np.all(done[:-1] == 0) and np.all(done[-1] == 1)
    full = oracle.PaperBatch(np.arange(n))
    oracle.paper_reset(m, full)
    oracle.paper_reset(m, full)
    assert np.array_equal(to_np(env.state).view(np.uint32),
                          full.state.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.params).view(np.uint32),
                          full.params.astype(np.float32).view(np.uint32))


def test_paper_bf16_value_over_trajectory_layout(oracle):
    torch = need_gpu()
    n, T = 1000, 5
    w = W.workload("paper_4096", n_envs=n)
    env = make_env(w, bias_std=0.1)
    obs = W.random_observations(6, T * n, dim=12).reshape(T, n, 12).transpose(0, 2, 1).copy()
    val = torch.empty((T, n), device="cuda")
    env.value(torch.from_numpy(obs).cuda(), val)
    vw = W.value_weights(w, 0.1)
    g = to_np(val)
    for t in (0, 2, 4):
        idx = np.r_[0, 1, 500, 999]
        ref = oracle.mlp(vw, 12, 256, 1, True, obs[t][:, idx].T.astype(np.float64))[:, 0]
        assert np.abs(g[t, idx] - ref).max() <= BF16_TOL
