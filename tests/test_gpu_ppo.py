"""GPU parity of the PPO learner's advantage estimation (env_gae) against the
oracle's plain recursion: random trajectories with episode ends at every
step length; the serial kernel (T <= 8 and T > 512) and each shape of the
chunked one (2 to 32 chunks of at most 8 or 16 steps, ragged last chunks,
an empty trailing chunk at T = 129, env counts off the 32-env block);
a real rollout's rewards, dones and values; and the argument checks."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import assert_close, make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu

GAE_TOL = 2e-5    # fp32 recursion of up to 128 terms vs float64


def _random_traj(seed, T, n, p_done=0.05):
    rng = np.random.Generator(np.random.Philox(key=[seed, 21]))
    rew = rng.normal(-1.0, 0.5, (T, n)).astype(np.float32)
    value = rng.normal(-20.0, 5.0, (T, n)).astype(np.float32)
    done = (rng.random((T, n)) < p_done).astype(np.uint8)
    last = rng.normal(-20.0, 5.0, n).astype(np.float32)
    return rew, done, value, last


@pytest.mark.parametrize("T,n,gamma,lam", [(128, 65536, 0.99, 0.95), (37, 999, 0.9, 0.8),
                                           (1, 300, 0.99, 0.95), (64, 4096, 1.0, 1.0),
                                           (20, 500, 0.99, 0.0), (16, 77, 0.99, 0.95),
                                           (8, 70, 0.99, 0.95), (9, 50, 0.99, 0.95),
                                           (17, 33, 0.99, 0.95), (129, 1000, 0.99, 0.95),
                                           (255, 65, 0.97, 0.9), (512, 96, 0.99, 0.95),
                                           (600, 40, 0.99, 0.95)])
def test_gae_matches_oracle(T, n, gamma, lam):
    torch = need_gpu()
    from oracle import ppo_oracle as P
    w = W.workload("ppo_65536", n_envs=n)
    env = make_env(w, policy=False)
    rew, done, value, last = _random_traj(T * 7 + n, T, n)
    dev = lambda a: torch.from_numpy(a).cuda()
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    env.gae(dev(rew), dev(done), dev(value), dev(last), gamma, lam, adv, ret)
    r_adv, r_ret = P.gae(rew, done, value, last, gamma, lam)
    scale = max(1.0, float(np.abs(r_ret).max()))
    assert_close(to_np(adv), r_adv, GAE_TOL, floor=scale, what="advantage")
    assert_close(to_np(ret), r_ret, GAE_TOL, floor=scale, what="return")


def test_gae_on_a_rollout():
    """The learner's input as produced: rewards, dones and values of a bf16
    rollout with episode ends inside the horizon, bootstrap value from the
    observation after the last step."""
    torch = need_gpu()
    from oracle import ppo_oracle as P
    n, T = 8192, 64
    w = W.workload("ppo_65536", n_envs=n, episode_len=40)
    env = make_env(w)
    env.reset()
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    obs = torch.empty((1, 18, n), device="cuda")
    env.observe(obs[0])
    last = torch.empty((1, n), device="cuda")
    env.value(obs, last)
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    env.gae(traj["rew"], traj["done"], traj["value"], last[0], 0.99, 0.95, adv, ret)
    assert to_np(traj["done"])[39].all()
    r_adv, r_ret = P.gae(to_np(traj["rew"]), to_np(traj["done"]), to_np(traj["value"]),
                         to_np(last[0]), 0.99, 0.95)
    scale = max(1.0, float(np.abs(r_ret).max()))
    assert_close(to_np(adv), r_adv, GAE_TOL, floor=scale, what="advantage")
    assert_close(to_np(ret), r_ret, GAE_TOL, floor=scale, what="return")


def test_gae_rejects_bad_arguments():
    torch = need_gpu()
    from paper_2512_13359_gb300 import auvenv
    n, T = 256, 4
    env = make_env(W.workload("ppo_65536", n_envs=n), policy=False)
    rew = torch.zeros((T, n), device="cuda")
    done = torch.zeros((T, n), dtype=torch.uint8, device="cuda")
    val = torch.zeros((T, n), device="cuda")
    last = torch.zeros(n, device="cuda")
    adv = torch.empty((T, n), device="cuda")
    ret = torch.empty((T, n), device="cuda")
    for g, l in ((1.5, 0.9), (0.9, -0.1), (float("nan"), 0.9)):
        with pytest.raises(auvenv.AuvError) as ei:
            env.gae(rew, done, val, last, g, l, adv, ret)
        assert ei.value.code == auvenv.AUV_ERR_INVALID
    with pytest.raises(auvenv.AuvError):
        env.gae(rew, done, val, last, 0.9, 0.9, rew, ret)      # adv aliases rew
    with pytest.raises(auvenv.AuvError):
        env.gae(rew, done, val, last, 0.9, 0.9, adv, adv)      # adv aliases ret
