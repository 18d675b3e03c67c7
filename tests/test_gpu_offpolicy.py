"""GPU parity of the off-policy pieces against their oracle: inverse
allocation (env_inverse_allocate) for feasible and saturating wrenches and
its round trip through the forward allocation; the replay buffer (rbuf_*):
every sampled slot index bit-exact and every sampled field equal to the
oracle ring's copy after inserts that wrap, a real rollout inserted at full
size with sampled rows checked against the trajectory, and rejections."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("n", [1, 1000, 65536])
def test_inverse_allocation_matches_oracle(n):
    torch = need_gpu()
    from oracle import offpolicy_oracle as F
    w = W.workload("ppo_65536", n_envs=64)
    env = make_env(w, policy=False)
    rng = np.random.default_rng(n)
    alloc = np.asarray(w["alloc"], dtype=np.float64).reshape(6, 8)
    u_true = rng.uniform(-1.3, 1.3, (8, n))                  # some infeasible
    tau = ((alloc * w["thrust_max"]) @ u_true).astype(np.float32)
    cmd = torch.empty((8, n), device="cuda")
    env.inverse_allocate(torch.from_numpy(tau).cuda(), cmd)
    got = to_np(cmd)
    ref = F.inverse_allocation(alloc, w["thrust_max"], tau.astype(np.float64))
    assert np.abs(got - ref).max() <= 2e-5
    assert np.all(np.abs(got) <= 1.0)
    feas = np.all(np.abs(ref) < 0.999, axis=0)
    if feas.any():
        back = (alloc * w["thrust_max"]) @ got[:, feas].astype(np.float64)
        scale = np.abs(tau[:, feas]).max()
        assert np.abs(back - tau[:, feas]).max() <= 2e-5 * scale


def _traj(rng, T, D, A, N):
    return (rng.normal(size=(T, D, N)).astype(np.float32),
            rng.normal(size=(T, A, N)).astype(np.float32),
            rng.normal(size=(T, N)).astype(np.float32),
            (rng.random((T, N)) < 0.1).astype(np.uint8),
            rng.normal(size=(D, N)).astype(np.float32))


@pytest.mark.parametrize("D,A,B", [(18, 8, 4099), (12, 6, 1), (12, 6, 63), (37, 5, 64),
                                   (37, 5, 4099)])
def test_replay_buffer_matches_oracle_ring(D, A, B):
    """Inserts that wrap a 1,000-slot ring, then samples checked field by
    field: the Fossen and paper widths and an odd width, batches of one, a
    partial and a whole 64-sample block, and a ragged 4,099."""
    torch = need_gpu()
    from oracle import offpolicy_oracle as F
    from paper_2512_13359_gb300 import auvenv
    C = 1000
    rb = auvenv.ReplayBuffer(D, A, C)
    ref = F.ReplayBuffer(D, A, C)
    rng = np.random.default_rng(1)
    dev = lambda x: torch.from_numpy(x).cuda()
    for T, N in ((3, 133), (2, 333), (1, 45)):                # the second insert wraps
        obs, act, rew, done, last = _traj(rng, T, D, A, N)
        rb.insert(dev(obs), dev(act), dev(rew), dev(done), dev(last))
        ref.insert(obs, act, rew, done, last)
        assert rb.size == (ref.size, ref.head)
    for draw in range(3):
        out = rb.sample(B, seed=77, draw=draw, with_idx=True)
        r = ref.sample(77, draw, B)
        assert np.array_equal(to_np(out["idx"]).view(np.uint32), r["idx"].astype(np.uint32))
        for k in ("obs", "act", "rew", "next_obs", "done"):
            assert np.array_equal(to_np(out[k]), r[k]), k


def test_replay_buffer_full_size_rollout():
    """A bf16 rollout of 65,536 envs x 16 steps inserted at once; 65,536
    samples checked against the trajectory arrays (slot s = t N + i)."""
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n, T = 65536, 16
    w = W.workload("ppo_65536", n_envs=n, episode_len=10)
    env = make_env(w)
    env.reset()
    traj = env.alloc_traj(T, keys=("obs", "act", "rew", "done"))
    env.rollout(T, traj)
    last = torch.empty((18, n), device="cuda")
    env.observe(last)
    rb = auvenv.ReplayBuffer(18, 8, 1 << 21)
    rb.insert(traj["obs"], traj["act"], traj["rew"], traj["done"], last)
    assert rb.size == (n * T, n * T)
    out = rb.sample(65536, seed=3, draw=0, with_idx=True)
    idx = to_np(out["idx"]).astype(np.int64)
    assert idx.max() < n * T and len(np.unique(idx)) > 60000
    t, i = idx // n, idx % n
    obs, act, rew, done = (to_np(traj[k]) for k in ("obs", "act", "rew", "done"))
    lo = to_np(last)
    assert np.array_equal(to_np(out["obs"]), obs[t, :, i])
    assert np.array_equal(to_np(out["act"]), act[t, :, i])
    assert np.array_equal(to_np(out["rew"]), rew[t, i])
    assert np.array_equal(to_np(out["done"]), done[t, i])
    nxt = np.where((t + 1 < T)[:, None], obs[np.minimum(t + 1, T - 1), :, i], lo[:, i].T)
    assert np.array_equal(to_np(out["next_obs"]), nxt)


def test_replay_buffer_rejects_bad_arguments():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    rb = auvenv.ReplayBuffer(18, 8, 100)
    with pytest.raises(auvenv.AuvError) as ei:
        rb.sample(10, 0, 0)                               # empty
    assert ei.value.code == auvenv.AUV_ERR_INVALID
    obs = torch.zeros((1, 18, 4))
    with pytest.raises(auvenv.AuvError) as ei:
        rb.insert(obs, torch.zeros((1, 8, 4)), torch.zeros((1, 4)),
                  torch.zeros((1, 4), dtype=torch.uint8), torch.zeros((18, 4)))
    assert ei.value.code == auvenv.AUV_ERR_SIZE          # host arrays
    with pytest.raises(auvenv.AuvError):
        auvenv.ReplayBuffer(18, 8, 0)
