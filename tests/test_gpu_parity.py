"""GPU parity through the C ABI against the CPU oracle: resets, Philox words
and done flags bit-exact; observation, action-replay dynamics and the fp32
closed-loop rollout within the fp32 tolerances; device status on injected
non-finite state; determinism of split rollouts."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import (REWARD_SUM_TOL, STATE_TOL, assert_close, make_env, need_gpu,
                         oracle_batch, to_np, u32)

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,n", [("tiny_64", 64), ("dr_16384", 16384), ("tiny_64", 1000)])
def test_reset_bit_exact(oracle, name, n):
    need_gpu()
    w = W.workload(name, n_envs=n)
    env = make_env(w, policy=False)
    env.reset()
    env.reset()          # second episode draw (episode index 1)
    m = oracle.model(w)
    ids = np.arange(n)
    b = oracle.Batch(ids)
    oracle.reset(m, b)
    oracle.reset(m, b)
    assert np.array_equal(to_np(env.state).view(np.uint32),
                          b.state.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.params).view(np.uint32),
                          b.params.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.t_ep), b.t_ep)
    assert np.array_equal(u32(env.episode), b.episode)


def test_masked_reset_touches_only_masked_envs(oracle):
    torch = need_gpu()
    w = W.workload("dr_16384", n_envs=300)
    env = make_env(w, policy=False)
    env.reset()
    before = to_np(env.state).copy()
    mask = torch.zeros(300, dtype=torch.uint8, device="cuda")
    mask[::7] = 1
    env.reset(mask)
    after = to_np(env.state)
    sel = np.zeros(300, bool)
    sel[::7] = True
    assert np.array_equal(after[:, ~sel], before[:, ~sel])
    m = oracle.model(w)
    b = oracle.Batch(np.arange(300)[sel])
    oracle.reset(m, b)
    oracle.reset(m, b)
    assert np.array_equal(after[:, sel].view(np.uint32), b.state.astype(np.float32).view(np.uint32))
    ep = u32(env.episode)
    assert np.all(ep[sel] == 2) and np.all(ep[~sel] == 1)


@pytest.mark.parametrize("stream_id,index,n_blocks", [(0, 0, 2), (0, (1 << 40) + 12345, 2),
                                                       (1, 3, 5), (1, 0xFFFFFFFF, 5)])
def test_philox_words_bit_exact(oracle, stream_id, index, n_blocks):
    torch = need_gpu()
    n = 4099
    w = W.workload("tiny_64", n_envs=n, seed=0xDEADBEEF)
    env = make_env(w, policy=False)
    out = torch.empty((4 * n_blocks, n), dtype=torch.int32, device="cuda")
    env.draw_words(stream_id, index, n_blocks, out)
    got = u32(out)
    for i in list(range(0, 40)) + [1000, 2047, 4095, 4098]:
        ref = np.concatenate([oracle.philox(i, 0xDEADBEEF, [index & 0xFFFFFFFF, index >> 32,
                                                             stream_id, b])
                              for b in range(n_blocks)])
        assert np.array_equal(got[:, i], ref), i


def _random_batch(rng, n):
    st = np.zeros((19, n), np.float32)
    pr = np.zeros((17, n), np.float32)
    st[0:3] = rng.uniform(-3, 3, (3, n))
    q = rng.standard_normal((4, n))
    st[3:7] = q / np.linalg.norm(q, axis=0)
    st[7:13] = rng.uniform(-1.5, 1.5, (6, n))
    st[13:19] = rng.uniform(-1.5, 1.5, (6, n))
    pr[0:3] = rng.uniform(-2, 2, (3, n))
    qd = rng.standard_normal((4, n))
    pr[3:7] = qd / np.linalg.norm(qd, axis=0)
    pr[7:10] = rng.uniform(0.8, 1.2, (3, n))
    pr[10] = rng.uniform(-2, 2, n)
    pr[11:14] = rng.uniform(-0.01, 0.01, (3, n))
    pr[14:17] = rng.uniform(-0.3, 0.3, (3, n))
    return st, pr


def test_observation_parity(oracle):
    torch = need_gpu()
    n = 1000
    w = W.workload("dr_16384", n_envs=n)
    env = make_env(w, policy=False)
    st, pr = _random_batch(np.random.default_rng(0), n)
    env.state.copy_(torch.from_numpy(st))
    env.params.copy_(torch.from_numpy(pr))
    out = torch.empty((18, n), dtype=torch.float32, device="cuda")
    env.observe(out)
    got = to_np(out)
    for i in range(0, n, 37):
        ref, _ = oracle.observe(st[:, i].astype(np.float64), pr[:, i].astype(np.float64))
        assert_close(got[:, i], ref, 2e-6, what=f"obs env {i}")


def _replay_compare(oracle, w, T, sample_ids, act_scale=0.7):
    torch = need_gpu()
    n = w["n_envs"]
    env = make_env(w, policy=False)
    env.reset()
    acts = W.replay_actions(5, T, n, act_scale)
    act_d = torch.from_numpy(acts).cuda()
    rew = torch.empty((T, n), dtype=torch.float32, device="cuda")
    done = torch.empty((T, n), dtype=torch.uint8, device="cuda")
    trace = torch.empty((T, 19, n), dtype=torch.float32, device="cuda")
    env.step_actions(act_d, rew, done, trace)
    assert env.status().code == 0
    m = oracle.model(w)
    ids = np.asarray(sample_ids)
    b = oracle_batch(oracle, m, ids)
    r_o, d_o, tr_o = oracle.replay(m, b, np.ascontiguousarray(acts[:, :, ids]), trace=True)
    g_tr = to_np(trace)[:, :, ids]
    g_rew = to_np(rew)[:, ids]
    g_done = to_np(done)[:, ids]
    assert np.array_equal(g_done, d_o)
    assert_close(g_tr, tr_o, STATE_TOL, what="state trace")
    assert_close(g_rew, r_o, STATE_TOL, what="per-step reward")
    H = min(100, T)
    assert_close(g_rew[:H].sum(0), r_o[:H].sum(0), REWARD_SUM_TOL, floor=1e-9,
                 what="reward sum over 100 steps")
    # steps that ended an episode carry the next episode's reset state exactly
    t_idx, e_idx = np.nonzero(d_o)
    if len(t_idx):
        exact = g_tr[t_idx, :, e_idx]
        assert np.array_equal(exact.astype(np.float32).view(np.uint32),
                              tr_o[t_idx, :, e_idx].astype(np.float32).view(np.uint32))
    final = to_np(env.state)[:, ids]
    assert_close(final, b.state, STATE_TOL, what="final state")
    return d_o


@pytest.mark.parametrize("name,n,T,L", [
    ("tiny_64", 64, 200, 500),
    ("fp32_4096", 4096, 200, 500),
    ("dr_16384", 16384, 150, 500),
    ("dr_16384", 999, 120, 37),          # ragged N, auto-resets inside the horizon
    ("ppo_65536", 65536, 128, 500),      # the benchmark's launch: 65,536 envs x 128 steps
])
def test_action_replay_parity(oracle, name, n, T, L):
    w = W.workload(name, n_envs=n, episode_len=L)
    rng = np.random.default_rng(1)
    ids = np.unique(np.r_[0, n - 1, rng.integers(0, n, 48)])
    d = _replay_compare(oracle, w, T, ids)
    if L < T:
        assert d.sum() > 0


def test_action_replay_saturated_thrust(oracle):
    """Commands far beyond the clip: every thruster saturates."""
    w = W.workload("dr_16384", n_envs=256)
    _replay_compare(oracle, w, 100, np.arange(0, 256, 5), act_scale=5.0)


def _rollout_compare(oracle, w, T, ids, horizon, bias_std=0.0):
    """Closed-loop fp32 rollout against the double oracle on sampled env ids.
    States are compared over `horizon` steps (closed-loop rounding growth
    bounds it), done flags over all T."""
    torch = need_gpu()
    env = make_env(w, bias_std=bias_std)
    env.reset()
    env.t_g = 77
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    assert env.status().code == 0
    assert env.t_g == 77 + T
    m = oracle.model(w)
    b = oracle_batch(oracle, m, ids)
    pw = W.policy_weights(w, bias_std)
    vw = W.value_weights(w, bias_std) if w["has_value"] else None
    out = oracle.rollout(m, b, pw, vw, 77, T)
    g = {k: to_np(v) for k, v in traj.items()}
    assert np.array_equal(g["done"][:, ids], out["done"])
    h = horizon
    assert_close(g["obs"][:h, :, ids], out["obs"][:h], STATE_TOL, what="obs")
    assert_close(g["act"][:h, :, ids], out["act"][:h], STATE_TOL, what="act")
    assert_close(g["logp"][:h, ids], out["logp"][:h], STATE_TOL, what="logp")
    assert_close(g["rew"][:h, ids], out["rew"][:h], STATE_TOL, what="rew")
    if "value" in g:
        assert_close(g["value"][:h, ids], out["value"][:h], STATE_TOL, what="value")
    H = min(100, T)
    assert_close(g["rew"][:H, ids].sum(0), out["rew"][:H].sum(0), REWARD_SUM_TOL, floor=1e-9,
                 what="reward sum")
    return env, g, out


@pytest.mark.parametrize("name,n,T,horizon", [
    ("tiny_64", 64, 200, 100),
    ("fp32_4096", 4096, 120, 100),
    ("dr_16384", 16384, 100, 100),
])
def test_fp32_rollout_parity(oracle, name, n, T, horizon):
    w = W.workload(name, n_envs=n)
    rng = np.random.default_rng(2)
    ids = np.unique(np.r_[0, n - 1, rng.integers(0, n, 24)])
    _rollout_compare(oracle, w, T, ids, horizon)


def test_fp32_rollout_with_value_and_logstd_head(oracle):
    """The 65,536-env workload's networks (policy with log-std head, value)
    evaluated in fp32, with non-zero biases exercising every bias path."""
    w = W.workload("ppo_65536", n_envs=2048, mlp="fp32")
    ids = np.r_[0, 5, 1000, 2047]
    _rollout_compare(oracle, w, 40, ids, 40, bias_std=0.1)


def test_auto_reset_state_bit_exact(oracle):
    """An episode that ends on the last step leaves the next episode's reset
    draw in the state buffers, bit for bit."""
    w = W.workload("dr_16384", n_envs=512, episode_len=10)
    env, g, out = _rollout_compare(oracle, w, 10, np.arange(0, 512, 17), 10)
    m = oracle.model(w)
    b = oracle.Batch(np.arange(512))
    oracle.reset(m, b)
    oracle.reset(m, b)
    assert np.all(g["done"][9] == 1)
    assert np.array_equal(to_np(env.state).view(np.uint32),
                          b.state.astype(np.float32).view(np.uint32))
    assert np.array_equal(to_np(env.params).view(np.uint32),
                          b.params.astype(np.float32).view(np.uint32))


def test_split_rollout_is_deterministic(oracle):
    """rollout(2T) equals rollout(T); rollout(T) bit for bit (state carried
    through HBM, noise stream indexed by the global step)."""
    torch = need_gpu()
    w = W.workload("dr_16384", n_envs=777, episode_len=23)
    e1 = make_env(w)
    e1.reset()
    t1 = e1.alloc_traj(40)
    e1.rollout(40, t1)
    e2 = make_env(w)
    e2.reset()
    ta = e2.alloc_traj(20)
    tb = e2.alloc_traj(20)
    e2.rollout(20, ta)
    e2.rollout(20, tb)
    for k in t1:
        joined = torch.cat([ta[k], tb[k]], 0)
        assert torch.equal(t1[k], joined), k
    assert torch.equal(e1.state, e2.state)


def test_checkpoint_resume_in_a_new_env(oracle):
    """Checkpoint = the caller's state, params and counter buffers plus the
    global step (env_get_step); restoring them into a fresh env (copy +
    env_set_step) continues the rollout bit for bit, trajectory and state."""
    torch = need_gpu()
    w = W.workload("dr_16384", n_envs=1000, episode_len=17)
    a = make_env(w)
    a.reset()
    a.rollout(25, a.alloc_traj(25))
    snap = {k: getattr(a, k).clone() for k in ("state", "params", "t_ep", "episode")}
    step = a.t_g
    assert step == 25
    b = make_env(w)
    for k, v in snap.items():
        getattr(b, k).copy_(v)
    b.t_g = step
    ta, tb = a.alloc_traj(30), b.alloc_traj(30)
    a.rollout(30, ta)
    b.rollout(30, tb)
    for k in ta:
        assert torch.equal(ta[k], tb[k]), k
    for k in snap:
        assert torch.equal(getattr(a, k), getattr(b, k)), k
    assert b.t_g == a.t_g == 55


@pytest.mark.parametrize("name,host", [("dr_16384", True), ("paper_4096", False)])
def test_snapshot_get_set_state(oracle, name, host):
    """env_get_state / env_set_state: a snapshot (state, params, t_ep,
    episode and the global step) taken mid-episode into page-locked host or
    device arrays, restored into a fresh env, continues bit for bit (the
    trajectory of the next launch, including resets inside it, and the final
    arrays); snapshots that do not fit the env are rejected."""
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n = 1000
    w = W.workload(name, n_envs=n, episode_len=17)
    a = make_env(w)
    a.reset()
    a.rollout(25, a.alloc_traj(25))
    snap = {k: (torch.empty(getattr(a, k).shape, dtype=getattr(a, k).dtype, pin_memory=True)
                if host else torch.empty_like(getattr(a, k)))
            for k in ("state", "params", "t_ep", "episode")}
    t_g = a.get_state(snap)
    torch.cuda.synchronize()
    assert t_g == 25 and snap["t_g"] == 25
    for k in ("state", "params", "t_ep", "episode"):
        assert torch.equal(snap[k].cuda(), getattr(a, k)), k
    b = make_env(w)
    b.set_state(snap)
    assert b.t_g == 25
    ta, tb = a.alloc_traj(30), b.alloc_traj(30)
    a.rollout(30, ta)
    b.rollout(30, tb)
    for k in ta:
        assert torch.equal(ta[k], tb[k]), k
    for k in ("state", "params", "t_ep", "episode"):
        assert torch.equal(getattr(a, k), getattr(b, k)), k
    # snapshots of another batch size or model, a bad header, a misaligned array
    c = make_env(dict(w, n_envs=n - 1))
    with pytest.raises(auvenv.AuvError) as e:
        c.set_state(snap)
    assert e.value.code == auvenv.AUV_ERR_INVALID
    other = W.workload("tiny_64" if W.is_paper(w) else "paper_tiny", n_envs=n)
    d = make_env(other, policy=False)
    with pytest.raises(auvenv.AuvError) as e:
        d.set_state(dict(snap, model=a.cfg.model))
    assert e.value.code == auvenv.AUV_ERR_INVALID
    with pytest.raises(auvenv.AuvError) as e:
        b.set_state(dict(snap, n_envs=n + 1))
    assert e.value.code == auvenv.AUV_ERR_INVALID
    raw = torch.empty(snap["t_ep"].numel() + 1, dtype=torch.int32, device="cuda")
    bad = dict(snap, t_ep=raw.view(torch.uint8)[1:])   # one byte past a 4-byte boundary
    with pytest.raises(auvenv.AuvError) as e:
        b.get_state(bad)
    assert e.value.code == auvenv.AUV_ERR_SIZE


def test_nan_state_is_reported(oracle):
    torch = need_gpu()
    w = W.workload("tiny_64", n_envs=300)
    env = make_env(w)
    env.reset()
    env.state[7, 123] = float("nan")
    env.state[8, 250] = float("inf")
    traj = env.alloc_traj(3, keys=("rew", "done"))
    env.rollout(3, traj)
    s = env.status()
    assert s.code == -5 and s.nan_flag == 1 and s.first_nan_env == 123
    env.clear_status()
    assert env.status().code == 0


def test_env_step_matches_rollout_row(oracle):
    torch = need_gpu()
    w = W.workload("tiny_64", n_envs=200)
    e1, e2 = make_env(w), make_env(w)
    e1.reset()
    e2.reset()
    obs = torch.empty((18, 200), device="cuda")
    rew = torch.empty((200,), device="cuda")
    done = torch.empty((200,), dtype=torch.uint8, device="cuda")
    e1.step(obs, rew, done)
    tr = e2.alloc_traj(1)
    e2.rollout(1, tr)
    assert torch.equal(obs, tr["obs"][0]) and torch.equal(rew, tr["rew"][0])
    assert torch.equal(done, tr["done"][0]) and torch.equal(e1.state, e2.state)


def test_pinned_host_trajectory(oracle):
    """Trajectory outputs in mapped page-locked host memory are written
    directly by the kernel and equal the device-buffer run."""
    torch = need_gpu()
    w = W.workload("tiny_64", n_envs=256)
    e1, e2 = make_env(w), make_env(w)
    e1.reset()
    e2.reset()
    td = e1.alloc_traj(15)
    th = e2.alloc_traj(15, pinned_host=True)
    e1.rollout(15, td)
    e2.rollout(15, th)
    torch.cuda.synchronize()
    for k in td:
        assert torch.equal(td[k].cpu(), th[k]), k


def test_invalid_buffers_rejected(oracle):
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    w = W.workload("tiny_64", n_envs=64)
    env = make_env(w)
    env.reset()
    unpinned = torch.empty((4, 64))          # pageable host memory
    with pytest.raises(auvenv.AuvError) as ei:
        env.rollout(4, {"rew": unpinned})
    assert ei.value.code == auvenv.AUV_ERR_SIZE
    with pytest.raises(auvenv.AuvError) as ei:
        env.rollout(0, {})
    assert ei.value.code == auvenv.AUV_ERR_INVALID
