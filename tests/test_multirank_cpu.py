"""The multi-GPU path on CPU: two gloo ranks each own a shard of global env
ids (paper_2512_13359_gb300.shard), step it with the oracle, and rank 0
checks that the shards together reproduce the unsharded batch bit for bit;
the timing reduction takes the slowest rank.  No GPU and no data-path
collective (the rollout's ranks exchange nothing)."""
import os
import socket

import numpy as np
import pytest

N_PER_RANK = 6
T = 12


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch.distributed as dist
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    from oracle import oracle as O
    from paper_2512_13359_gb300 import shard, workloads as W
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        base, n = shard.env_range(rank, N_PER_RANK)
        w = W.workload("ppo_65536", n_envs=n, episode_len=5)
        m = O.model(w)
        b = O.Batch(np.arange(base, base + n))
        O.reset(m, b)
        out = O.rollout(m, b, W.policy_weights(w), W.value_weights(w), 0, T)
        slowest = shard.max_over_ranks(1.0 + rank, dist)
        shard.barrier(dist)
        np.savez(os.path.join(out_dir, f"rank{rank}.npz"), state=b.state, rew=out["rew"],
                 done=out["done"], obs=out["obs"], slowest=slowest, base=base)
    finally:
        dist.destroy_process_group()


def test_two_rank_shards_reproduce_the_batch(tmp_path, oracle):
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    world = 2
    mp.spawn(_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    from paper_2512_13359_gb300 import workloads as W
    w = W.workload("ppo_65536", n_envs=world * N_PER_RANK, episode_len=5)
    m = oracle.model(w)
    b = oracle.Batch(np.arange(world * N_PER_RANK))
    oracle.reset(m, b)
    full = oracle.rollout(m, b, W.policy_weights(w), W.value_weights(w), 0, T)
    parts = [np.load(tmp_path / f"rank{r}.npz") for r in range(world)]
    assert [int(p["base"]) for p in parts] == [0, N_PER_RANK]
    assert np.array_equal(np.concatenate([p["state"] for p in parts], axis=1), b.state)
    assert np.array_equal(np.concatenate([p["rew"] for p in parts], axis=1), full["rew"])
    assert np.array_equal(np.concatenate([p["done"] for p in parts], axis=1), full["done"])
    assert np.array_equal(np.concatenate([p["obs"] for p in parts], axis=2), full["obs"])
    assert all(float(p["slowest"]) == 2.0 for p in parts)


def test_env_range_validation():
    from paper_2512_13359_gb300 import shard
    assert shard.env_range(3, 100) == (300, 100)
    with pytest.raises(ValueError):
        shard.env_range(-1, 10)
    with pytest.raises(ValueError):
        shard.env_range(1 << 22, 1 << 11)
    assert shard.max_over_ranks(3.5) == 3.5


# ---------------------------------------------------------------------------
# The learner's exchange: data-parallel PPO (gradient averaged over ranks).
# ---------------------------------------------------------------------------
LEARN_STEPS = 3


def _rank_traj(rank, T=4, N=50, D=18, A=8):
    rng = np.random.default_rng(100 + rank)
    return dict(obs=rng.normal(size=(T, D, N)), act=rng.normal(size=(T, A, N)),
                logp=rng.normal(size=(T, N)) - 10.0, adv=rng.normal(size=(T, N)),
                ret=rng.normal(size=(T, N)))


def _learner_worker(rank, world, port, out_dir):
    import torch
    import torch.distributed as dist
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    from oracle import ppo_oracle as P
    from paper_2512_13359_gb300 import shard, workloads as W
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        D, H, A = 18, 16, 8
        pw = W.mlp_weights(0, D, H, 2 * A, 0, 0.1)
        vw = W.mlp_weights(0, D, H, 1, 1, 0.1)
        hp = dict(clip_eps=0.2, vf_coef=0.5, ent_coef=0.01, max_grad_norm=0.5, lr=1e-3,
                  adam_beta1=0.9, adam_beta2=0.999, adam_eps=1e-8, logstd_min=-5.0,
                  logstd_max=2.0, norm_adv=True)
        L = P.Learner(pw, vw, (D, H, A), hp, seed=9)
        traj = _rank_traj(rank)
        for j in range(LEARN_STEPS):
            _, g = L.grads(traj, 0, j, 64)
            gt = torch.from_numpy(g.copy())
            shard.mean_over_ranks(gt, dist)
            L.apply(gt.numpy())
        np.save(os.path.join(out_dir, f"learner{rank}.npy"), L.w)
    finally:
        dist.destroy_process_group()


def test_two_rank_learner_averages_gradients(tmp_path):
    """Two gloo ranks, each with its own trajectory, average every
    minibatch gradient and take the same Adam step: both end with identical
    weights, equal to one process applying the mean of the two gradients."""
    pytest.importorskip("torch")
    import torch.multiprocessing as mp
    from oracle import ppo_oracle as P
    from paper_2512_13359_gb300 import workloads as W
    world = 2
    mp.spawn(_learner_worker, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    w0, w1 = (np.load(tmp_path / f"learner{r}.npy") for r in range(world))
    assert np.array_equal(w0, w1)
    D, H, A = 18, 16, 8
    hp = dict(clip_eps=0.2, vf_coef=0.5, ent_coef=0.01, max_grad_norm=0.5, lr=1e-3,
              adam_beta1=0.9, adam_beta2=0.999, adam_eps=1e-8, logstd_min=-5.0,
              logstd_max=2.0, norm_adv=True)
    pw = W.mlp_weights(0, D, H, 2 * A, 0, 0.1)
    vw = W.mlp_weights(0, D, H, 1, 1, 0.1)
    ref = [P.Learner(pw, vw, (D, H, A), hp, seed=9) for _ in range(world)]
    trajs = [_rank_traj(r) for r in range(world)]
    for j in range(LEARN_STEPS):
        gs = [L.grads(t, 0, j, 64)[1] for L, t in zip(ref, trajs)]
        mean = (gs[0] + gs[1]) / 2
        for L in ref:
            L.apply(mean)
    assert np.allclose(w0, ref[0].w, rtol=1e-12, atol=1e-15)
    assert not np.allclose(w0, P.Learner(pw, vw, (D, H, A), hp, seed=9).w)
