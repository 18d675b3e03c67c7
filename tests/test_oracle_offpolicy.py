"""Pins for the oracle of inverse allocation and the replay buffer:
B (F_max u) = tau for feasible wrenches, minimum norm (equal to the SVD
least-squares solution and orthogonal to B's null space), saturation for
infeasible ones and a hand example; the ring's slot arithmetic, next
observations and overwrite order on a hand-checked case; the sample
indices against the top bits of Philox for power-of-two sizes, their range,
spread and determinism."""
import numpy as np
import pytest

from oracle import oracle as O
from oracle import offpolicy_oracle as F
from paper_2512_13359_gb300 import workloads as W


def test_inverse_allocation_solves_feasible_wrenches():
    w = W.workload("ppo_65536")
    alloc = np.asarray(w["alloc"], dtype=np.float64).reshape(6, 8)
    rng = np.random.default_rng(0)
    u_true = rng.uniform(-0.4, 0.4, (8, 50))
    tau = (alloc * w["thrust_max"]) @ u_true
    u = F.inverse_allocation(alloc, w["thrust_max"], tau)
    assert np.allclose((alloc * w["thrust_max"]) @ u, tau, rtol=1e-10, atol=1e-9)
    lsq = np.linalg.lstsq(alloc * w["thrust_max"], tau, rcond=None)[0]
    assert np.allclose(u, lsq, rtol=1e-9, atol=1e-12)
    null = np.linalg.svd(alloc)[2][6:]            # 2 x 8 basis of B's null space
    assert np.abs(null @ u).max() < 1e-12
    assert np.all(np.linalg.norm(u, axis=0) <= np.linalg.norm(u_true, axis=0) + 1e-12)


def test_inverse_allocation_saturates_and_hand_case():
    alloc = np.hstack([np.eye(6), np.zeros((6, 2))])
    tau = np.array([[5.0], [-50.0], [0.0], [20.0], [-19.0], [1.0]])
    u = F.inverse_allocation(alloc, 20.0, tau)
    assert np.allclose(u[:, 0], [0.25, -1.0, 0.0, 1.0, -0.95, 0.05, 0.0, 0.0], atol=1e-15)
    w = W.workload("ppo_65536")
    big = np.full((6, 3), 1e4)
    u = F.inverse_allocation(w["alloc"], w["thrust_max"], big)
    assert np.all(np.abs(u) <= 1.0) and np.any(np.abs(u) == 1.0)


def test_ring_buffer_slots_and_next_observations():
    rb = F.ReplayBuffer(2, 1, 5)
    T, N = 2, 2
    obs = np.arange(T * 2 * N, dtype=np.float32).reshape(T, 2, N)     # obs[t][k][i]
    act = -np.arange(T * N, dtype=np.float32).reshape(T, 1, N)
    rew = np.array([[1, 2], [3, 4]], np.float32)
    done = np.array([[0, 1], [0, 0]], np.uint8)
    last = np.array([[100, 101], [102, 103]], np.float32)
    rb.insert(obs, act, rew, done, last)
    assert (rb.head, rb.size) == (4, 4)
    # slot 1 = (t 0, env 1): obs[0][:,1] = (1, 3), next = obs[1][:,1] = (5, 7)
    assert np.array_equal(rb.obs[1], [1, 3]) and np.array_equal(rb.next_obs[1], [5, 7])
    assert rb.done[1] == 1 and rb.rew[1] == 2 and rb.act[1, 0] == -1
    # slot 3 = (t 1, env 1): next = last_obs[:,1] = (101, 103)
    assert np.array_equal(rb.next_obs[3], [101, 103])
    rb.insert(obs, act, rew + 10, done, last)      # 4 more: slots 4, 0, 1, 2
    assert (rb.head, rb.size) == (3, 5)
    assert rb.rew[4] == 11 and rb.rew[0] == 12 and rb.rew[2] == 14 and rb.rew[3] == 4


def test_sample_indices_definition_and_spread():
    seed, draw = 12345, 7
    for k in (0, 1, 5, 16):
        size = 1 << k
        idx = O.rbuf_indices(seed, draw, size, 64)
        for b in (0, 1, 63):
            word = O.philox(seed & 0xFFFFFFFF, seed >> 32, [b, 0x52420000, draw, 0])[0]
            assert idx[b] == (int(word) >> (32 - k) if k else 0)
    idx = O.rbuf_indices(seed, draw, 1000, 100000)
    assert idx.max() < 1000
    counts = np.bincount(idx, minlength=1000)
    chi2 = ((counts - 100) ** 2 / 100).sum()
    assert 800 < chi2 < 1200                       # 999 degrees of freedom
    assert np.array_equal(idx, O.rbuf_indices(seed, draw, 1000, 100000))
    assert not np.array_equal(idx, O.rbuf_indices(seed, draw + 1, 1000, 100000))
