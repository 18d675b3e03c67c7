"""TEST INFRASTRUCTURE: the oracle of the PPO learner's on-GPU pieces
(paper §III-A: PPO with its clipped surrogate objective, Schulman et al.
2017).  Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline /
reference legs may import this module; it shares nothing with the CUDA
library.  Plain numpy in float64.

Generalised advantage estimation (Schulman, Moritz, Levine, Jordan, Abbeel,
"High-dimensional continuous control using generalized advantage
estimation", ICLR 2016), over a trajectory in the rollout's layout
[T][N] (step t of env i at t*N + i):

  delta_t = r_t + gamma (1 - d_t) V_{t+1} - V_t,   V_T = bootstrap value
  A_t     = delta_t + gamma lambda (1 - d_t) A_{t+1},  A_T = 0
  R_t     = A_t + V_t                              (the value target)

d_t = 1 marks the last step of an episode: nothing of the next episode (its
reset state's value, its rewards) flows back across it.
"""
from __future__ import annotations

import numpy as np


def gae(rew, done, value, last_value, gamma: float, lam: float):
    """Advantages and returns [T][N] (float64) by the backward recursion."""
    rew = np.asarray(rew, dtype=np.float64)
    value = np.asarray(value, dtype=np.float64)
    nonterm = 1.0 - np.asarray(done, dtype=np.float64)
    T, n = rew.shape
    adv = np.zeros((T, n))
    a_next = np.zeros(n)
    v_next = np.asarray(last_value, dtype=np.float64)
    for t in range(T - 1, -1, -1):
        delta = rew[t] + gamma * nonterm[t] * v_next - value[t]
        a_next = delta + gamma * lam * nonterm[t] * a_next
        adv[t] = a_next
        v_next = value[t]
    return adv, adv + value
