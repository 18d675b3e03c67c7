"""Failure detection on the GPU without faulting it: a bounded device wait is
made to run out (a barrier phase nothing completes), the kernel returns, the
timeout is reported through env_status, and the context keeps working."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from parity_util import make_env, need_gpu, to_np

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_reports():
    torch = need_gpu()
    import time
    w = W.workload("ppo_65536", n_envs=512)
    env = make_env(w)
    env.reset()
    t0 = time.perf_counter()
    env.selftest_wait_timeout(20000)          # 20 ms
    st = env.status()
    dt = time.perf_counter() - t0
    assert st.code == -4 and st.timeouts == 1
    assert 0.015 < dt < 5.0
    # the context is still usable: clear and run a rollout
    env.clear_status()
    traj = env.alloc_traj(4)
    env.rollout(4, traj)
    st = env.status()
    assert st.code == 0 and st.timeouts == 0
    assert np.all(np.isfinite(to_np(traj["rew"])))


def test_selftest_rejects_bad_limits():
    need_gpu()
    from paper_2512_13359_gb300 import auvenv
    env = make_env(W.workload("tiny_64"), policy=False)
    with pytest.raises(auvenv.AuvError):
        env.selftest_wait_timeout(0)
    with pytest.raises(auvenv.AuvError):
        env.selftest_wait_timeout(10 ** 7)
