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
    in windows of 64 steps: the same rollout run as launches of 64 steps is
    bit-identical to the single launch, and its state at each window start
    restarts the oracle (fp32 against double rounding drift can reach the
    1e-5 tolerance within about a hundred steps)."""
    torch = need_gpu()
    w = W.workload("paper_4096", n_envs=n, episode_len=L)
    traj, final = _run(w, T)
    resync = None
    if T > 64:
        env = make_env(w)
        env.reset()
        resync, parts = {}, []
        for t0 in range(0, T, 64):
            resync[t0] = (to_np(env.state), to_np(env.params), to_np(env.t_ep),
                          to_np(env.episode))
            part = env.alloc_traj(min(64, T - t0))
            env.rollout(min(64, T - t0), part)
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


# fp32 networks on the tensor cores (kind::tf32).  Weights, observations and
# hidden activations are rounded to tf32 (10 explicit mantissa bits, relative
# error below 2^-11), tanh is the hardware approximation (about 2^-11) and
# sums are fp32: each hidden unit is within about 2^-10 of its exact value
# relative to its size, and with N(0, 1/fan_in) weights these errors add in
# quadrature through the 256-wide layers to a few 1e-4 on outputs of order
# one.  TF32_TOL bounds them with a margin against the oracle's exact (double)
# network; the measured maximum is printed.
TF32_TOL = 3e-3


def _windows(w, T, win=16):
    """Run T steps as one launch and as launches of `win` steps; the two must
    agree bit for bit, and the windowed run gives the state at each window
    start for the checker to restart the oracle from.  The tolerance is on
    the state one step produces (1e-5 relative); over tens of steps fp32 and
    double rounding compound (with this workload's unit action noise the
    thrust saturates often and the attitude error grows fastest: 1.1e-5 on
    one env's body-frame position 32 steps after a common state), so
    windows of 16 steps keep the comparison about single steps."""
    torch = need_gpu()
    traj, final = _run(w, T)
    env = make_env(w)
    env.reset()
    resync, parts = {}, []
    for t0 in range(0, T, win):
        resync[t0] = (to_np(env.state), to_np(env.params), to_np(env.t_ep), to_np(env.episode))
        part = env.alloc_traj(min(win, T - t0))
        env.rollout(min(win, T - t0), part)
        parts.append(part)
    assert env.status().code == 0
    for k in traj:
        assert torch.equal(torch.cat([p[k] for p in parts]), traj[k]), k
    return traj, final, resync


@pytest.mark.parametrize("name,n,T,L", [("fp32_4096", 4096, 1000, 500),
                                        ("dr_16384", 16384, 1000, 500),
                                        ("fp32_4096", 999, 50, 17),
                                        ("dr_16384", 300, 20, 6)])
def test_tf32_engine_rollout_every_step(oracle, name, n, T, L):
    """The fp32 workloads' tensor-core rollout (k_rollout_tf32): 4,096 envs x
    1,000 steps (the paper's env count) and 16,384 envs x 1,000 steps with
    domain randomisation and current, both with auto-resets at step 500, plus ragged sizes that reset
    inside short launches; every step of 40 sampled envs against the oracle."""
    need_gpu()
    w = W.workload(name, n_envs=n, episode_len=L, mlp="tf32")
    traj, final, resync = _windows(w, T) if T > 16 else (*_run(w, T), None)
    ids = sample_ids(n, k=40)
    worst = check_engine_rollout(oracle, w, traj, ids, T, final_state=final, resync=resync,
                                 net_tol=TF32_TOL)
    print(f"[tf32 engine {name} n={n} T={T} L={L}] " +
          " ".join(f"{k} {v:.2e}" for k, v in worst.items()))
    assert worst["act"] <= TF32_TOL


@pytest.mark.parametrize("seed", [1, 2])
def test_tf32_engine_rollout_other_seeds(oracle, seed):
    """The paper evaluates its 4,096-env training at three seeds (§V-A1,
    Fig. 2); the second workload carries seeds 0, 1 and 2.  Seed 0 runs the
    full 1,000 steps above; seeds 1 and 2 (other reset draws, goals and
    action noise for every env) run 64 steps at the full 4,096 envs, every
    step of 40 sampled envs against the oracle."""
    need_gpu()
    w = W.workload("fp32_4096", n_envs=4096, episode_len=500, mlp="tf32", seed=seed)
    T = 64
    traj, final, resync = _windows(w, T)
    ids = sample_ids(4096, k=40, seed=seed)
    worst = check_engine_rollout(oracle, w, traj, ids, T, final_state=final, resync=resync,
                                 net_tol=TF32_TOL)
    print(f"[tf32 engine fp32_4096 seed={seed}] " +
          " ".join(f"{k} {v:.2e}" for k, v in worst.items()))
    assert worst["act"] <= TF32_TOL
