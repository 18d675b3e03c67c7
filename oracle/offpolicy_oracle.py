"""TEST INFRASTRUCTURE: the oracle of the deployment and off-policy pieces.
Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline /
reference legs may import this module; it shares nothing with the CUDA
library.  Plain numpy in float64 (the replay buffer stores float32 as the
library does, since it copies and does no arithmetic).

Inverse allocation (paper §V-B: the controllers' body-frame wrench is mapped
to thruster commands through the allocation matrix): with B the 6 x 8
allocation matrix and F_max the thrust limit, the commands are the
minimum-norm solution of B (F_max u) = tau, clipped to the thrusters' range,
    u = clip(pinv(F_max B) tau, -1, 1).

DroQ replay buffer (paper §III-A, off-policy learning from replayed
experience; Hiraoka et al. 2022): a ring of `capacity` transitions
(obs, act, rew, next_obs, done).  Inserting a rollout's trajectory of T steps
x N envs writes transition (t, i) at slot (head + t*N + i) mod capacity with
next_obs = obs[t+1] (last_obs for t = T-1); a sample draws indices uniformly
from [0, size) by the counter-based generator of oracle.rbuf_indices.
"""
from __future__ import annotations

import numpy as np


def inverse_allocation(alloc, thrust_max: float, wrench):
    """alloc [6][8], wrench [6][n] -> commands [8][n] (float64)."""
    Bm = np.asarray(alloc, dtype=np.float64).reshape(6, 8) * float(thrust_max)
    u = np.linalg.pinv(Bm) @ np.asarray(wrench, dtype=np.float64)
    return np.clip(u, -1.0, 1.0)


class ReplayBuffer:
    def __init__(self, obs_dim: int, act_dim: int, capacity: int):
        self.D, self.A, self.C = obs_dim, act_dim, capacity
        self.obs = np.zeros((capacity, obs_dim), np.float32)
        self.act = np.zeros((capacity, act_dim), np.float32)
        self.rew = np.zeros(capacity, np.float32)
        self.next_obs = np.zeros((capacity, obs_dim), np.float32)
        self.done = np.zeros(capacity, np.uint8)
        self.head = 0
        self.size = 0

    def insert(self, obs, act, rew, done, last_obs):
        """obs [T][D][N], act [T][A][N], rew / done [T][N], last_obs [D][N]."""
        T, D, N = obs.shape
        for t in range(T):
            nxt = obs[t + 1] if t + 1 < T else last_obs
            for i in range(N):
                s = (self.head + t * N + i) % self.C
                self.obs[s] = obs[t, :, i]
                self.act[s] = act[t, :, i]
                self.rew[s] = rew[t, i]
                self.next_obs[s] = nxt[:, i]
                self.done[s] = done[t, i]
        self.head = (self.head + T * N) % self.C
        self.size = min(self.size + T * N, self.C)

    def sample(self, seed: int, draw: int, B: int):
        from oracle import oracle as O
        idx = O.rbuf_indices(seed, draw, self.size, B).astype(np.int64)
        return dict(idx=idx, obs=self.obs[idx], act=self.act[idx], rew=self.rew[idx],
                    next_obs=self.next_obs[idx], done=self.done[idx])
