"""Every step of the tensor-core (bf16, tcgen05) rollout against the oracle,
at the launch sizes the benchmark times and at ragged sizes with
auto-resets inside the launch (tests/engine_check.py: the oracle replays
the kernel's own actions for the physics, and evaluates its own bf16
networks, log-std clamp and normals on the kernel's observations for the
draw and the value)."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from engine_check import check_engine_rollout, sample_ids
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu


def _run(w, T):
    env = make_env(w)
    env.reset()
    traj = env.alloc_traj(T)
    env.rollout(T, traj)
    st = env.status()
    assert st.code == 0, (st.code, st.timeouts)
    final = (to_np(env.state), to_np(env.params), to_np(env.t_ep), to_np(env.episode))
    return traj, final


@pytest.mark.parametrize("n,T,L", [(65536, 128, 500), (1000, 40, 17), (300, 9, 4),
                                   (16384, 30, 11)])
def test_engine_rollout_every_step_fossen(oracle, n, T, L):
    """The Fossen model's fused rollout (k_engine, SIM = 0).  65,536 x 128 is
    the benchmark's launch; the ragged cases end episodes inside the launch,
    so auto-resets and the post-reset draws are checked mid-trajectory."""
    need_gpu()
    w = W.workload("ppo_65536", n_envs=n, episode_len=L)
    traj, final = _run(w, T)
    ids = sample_ids(n, k=40)
    worst = check_engine_rollout(oracle, w, traj, ids, T, final_state=final)
    print(f"[engine fossen n={n} T={T} L={L}] " +
          " ".join(f"{k} {v:.2e}" for k, v in worst.items()))


@pytest.mark.parametrize("n,T,L", [(4096, 512, 512), (999, 60, 23), (5000, 20, 7)])
def test_engine_rollout_every_step_paper(oracle, n, T, L):
    """The paper model's fused rollout (k_engine, SIM = 1).  4,096 x 512 is
    the benchmark's launch (the paper's env count and episode length,
    §IV-A, §V-A1); the ragged cases reset inside the launch, clearing the
    action history of Eq. 7's moving average.  The long launch is checked
    in windows of 128 steps: the same rollout run as four launches of 128
    steps is bit-identical to the single launch, and its state at each
    window start restarts the oracle (fp32 against double rounding drift
    reaches the 1e-5 tolerance after about 400 steps)."""
    torch = need_gpu()
    w = W.workload("paper_4096", n_envs=n, episode_len=L)
    traj, final = _run(w, T)
    resync = None
    if T > 128:
        env = make_env(w)
        env.reset()
        resync, parts = {}, []
        for t0 in range(0, T, 128):
            resync[t0] = (to_np(env.state), to_np(env.params), to_np(env.t_ep),
                          to_np(env.episode))
            part = env.alloc_traj(min(128, T - t0))
            env.rollout(min(128, T - t0), part)
            parts.append(part)
        assert env.status().code == 0
        for k in ("obs", "act", "logp", "rew", "done"):
            assert torch.equal(torch.cat([p[k] for p in parts]), traj[k]), k
    ids = sample_ids(n, k=40)
    worst = check_engine_rollout(oracle, w, traj, ids, T, final_state=final, resync=resync)
    print(f"[engine paper n={n} T={T} L={L}] " +
          " ".join(f"{k} {v:.2e}" for k, v in worst.items()))


def test_engine_rollout_every_step_after_a_first_launch(oracle):
    """A second launch continues the first: global step t_g0 = T1, state
    carried in the caller's buffers, noise of the later steps."""
    need_gpu()
    n, T1, T2 = 2000, 13, 21
    w = W.workload("ppo_65536", n_envs=n, episode_len=9)
    env = make_env(w)
    env.reset()
    t1 = env.alloc_traj(T1)
    env.rollout(T1, t1)
    t2 = env.alloc_traj(T2)
    env.rollout(T2, t2)
    assert env.status().code == 0
    full = {k: np.concatenate([to_np(t1[k]), to_np(t2[k])]) for k in t1}
    final = (to_np(env.state), to_np(env.params), to_np(env.t_ep), to_np(env.episode))
    ids = sample_ids(n, k=40)
    check_engine_rollout(oracle, w, full, ids, T1 + T2, final_state=final)
