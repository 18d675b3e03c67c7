"""env_rollout with page-locked host trajectory arrays: the library runs the
steps in segments through device staging buffers and copies each segment to
the host arrays while the next one computes.  Where the arrays live must not
change a single bit: these tests compare host, device and mixed placements
of the same rollout, including a ragged last segment, a second call that
reuses the staging buffers, and the value pass fed from staged observations.
"""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu

KEYS = ("obs", "act", "logp", "value", "rew", "done")


def _run(w, T, placement, calls=2):
    """Rollouts of T steps; placement maps each key to 'host' or 'device'."""
    import torch
    env = make_env(w)
    env.reset()
    outs = []
    for _ in range(calls):
        traj = {}
        for k in KEYS:
            dev = env.alloc_traj(T, keys=(k,), pinned_host=placement[k] == "host")
            traj.update(dev)
        env.rollout(T, traj)
        torch.cuda.synchronize()
        outs.append({k: to_np(v).copy() for k, v in traj.items()})
    assert env.status().code == 0
    state = to_np(env.state).copy()
    return outs, state


@pytest.mark.parametrize("n,T", [(65536, 37), (1000, 9)])
def test_host_trajectory_matches_device(n, T):
    """65,536 envs x 37 steps runs as segments of 8, 8, 8, 8, 5 (each staging
    buffer used three or two times); 1,000 envs x 9 steps is a single
    segment."""
    need_gpu()
    w = W.workload("ppo_65536", n_envs=n)
    dev_out, dev_state = _run(w, T, {k: "device" for k in KEYS})
    host_out, host_state = _run(w, T, {k: "host" for k in KEYS})
    mixed = {"obs": "device", "act": "host", "logp": "device", "value": "host", "rew": "host",
             "done": "device"}
    mix_out, mix_state = _run(w, T, mixed)
    for c in range(2):
        for k in KEYS:
            assert np.array_equal(dev_out[c][k], host_out[c][k]), (c, k)
            assert np.array_equal(dev_out[c][k], mix_out[c][k]), (c, k)
    assert np.array_equal(dev_state, host_state)
    assert np.array_equal(dev_state, mix_state)
    # the second call continued the first (new observations, same env count)
    assert not np.array_equal(dev_out[0]["obs"], dev_out[1]["obs"])


def test_host_single_step_written_in_place():
    """T = 1 with host arrays (env_step) writes through the device mapping."""
    torch = need_gpu()
    w = W.workload("ppo_65536", n_envs=4096)
    a, b = make_env(w), make_env(w)
    a.reset()
    b.reset()
    obs_d = torch.empty((1, 18, 4096), device="cuda")
    rew_d = torch.empty((1, 4096), device="cuda")
    done_d = torch.empty((1, 4096), dtype=torch.uint8, device="cuda")
    obs_h = torch.empty((1, 18, 4096), pin_memory=True)
    rew_h = torch.empty((1, 4096), pin_memory=True)
    done_h = torch.empty((1, 4096), dtype=torch.uint8, pin_memory=True)
    for _ in range(3):
        a.step(obs_d, rew_d, done_d)
        b.step(obs_h, rew_h, done_h)
        torch.cuda.synchronize()
        assert np.array_equal(to_np(obs_d), obs_h.numpy())
        assert np.array_equal(to_np(rew_d), rew_h.numpy())
        assert np.array_equal(to_np(done_d), done_h.numpy())
