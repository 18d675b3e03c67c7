"""The every-step rollout checker (tests/engine_check.py) on the CPU: the
oracle's own bf16 rollout passes it for both models, with auto-resets inside
the horizon, and a single wrong value in any checked array fails it."""
import numpy as np
import pytest

from paper_2512_13359_gb300 import workloads as W
from engine_check import check_engine_rollout, sample_ids


def _oracle_traj(oracle, w, T, ids):
    """The oracle's rollout of the envs `ids`, placed at their columns of
    full-width [T][K][N] arrays (the other columns zero)."""
    paper = W.is_paper(w)
    n = int(w["n_envs"])
    m = oracle.paper_model(w) if paper else oracle.model(w)
    b = oracle.PaperBatch(ids) if paper else oracle.Batch(ids)
    (oracle.paper_reset if paper else oracle.reset)(m, b)
    roll = oracle.paper_rollout if paper else oracle.rollout
    part = roll(m, b, W.policy_weights(w), W.value_weights(w), 0, T)
    out = {}
    for k, v in part.items():
        full = np.zeros(v.shape[:-1] + (n,), dtype=v.dtype)
        full[..., ids] = v
        out[k] = full
    final = []
    for v in (b.state, b.params, b.t_ep, b.episode):
        full = np.zeros(v.shape[:-1] + (n,), dtype=v.dtype)
        full[..., ids] = v
        final.append(full)
    return out, tuple(final)


@pytest.mark.parametrize("name", ["ppo_65536", "paper_4096"])
def test_checker_accepts_the_oracle_rollout(oracle, name):
    T = 12
    w = W.workload(name, n_envs=200, episode_len=5)
    ids = sample_ids(200, k=8)
    out, final = _oracle_traj(oracle, w, T, ids)
    assert out["done"][4][ids].all() and out["done"][9][ids].all()
    worst = check_engine_rollout(oracle, w, out, ids, T, final_state=final)
    assert worst["act"] < 1e-6 and worst["value"] < 1e-9 and worst["rew"] < 1e-6


@pytest.mark.parametrize("key,t,delta", [("rew", 3, 2e-3), ("act", 6, 0.05), ("logp", 1, 0.2),
                                         ("value", 7, 0.02), ("obs", 10, 1e-3),
                                         ("done", 2, 1)])
def test_checker_rejects_a_planted_error(oracle, key, t, delta):
    T = 12
    w = W.workload("ppo_65536", n_envs=200, episode_len=5)
    ids = sample_ids(200, k=8)
    out, final = _oracle_traj(oracle, w, T, ids)
    j = int(ids[3])
    bad = {k: v.copy() for k, v in out.items()}
    if key == "done":
        bad["done"][t, j] ^= 1
    elif bad[key].ndim == 3:
        bad[key][t, 0, j] += delta
    else:
        bad[key][t, j] += delta
    with pytest.raises(AssertionError):
        check_engine_rollout(oracle, w, bad, ids, T, final_state=final)
