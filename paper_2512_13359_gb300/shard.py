"""Multi-GPU sharding of the batched rollout.

Environments are independent (paper §IV-A: every env evolves on its own,
with its own initial conditions and randomisation), so one process per GPU
owns a contiguous range of global env ids and ranks exchange nothing on the
data path.  Local env i of rank r is global env r * n + i; its Philox streams
are keyed by the global id (auv_config.env_id_base), so any sharding of a
batch reproduces the unsharded batch exactly.  torch.distributed is used only
to align ranks and to take the slowest rank's time.

The learner is the one place with an exchange: a data-parallel PPO update
computes each rank's minibatch gradient (ppo_grads, a flat parameter
vector), averages the vectors over ranks (mean_over_ranks, one all-reduce
per gradient step) and takes the same Adam step everywhere (ppo_apply with
the averaged vector), so every rank's weights stay identical.
"""
from __future__ import annotations

import os


def world():
    """(rank, world_size, local_rank) from the torchrun environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def env_range(rank: int, n_per_rank: int) -> tuple[int, int]:
    """Global id of this rank's first env and its env count (weak scaling:
    every rank owns n_per_rank envs)."""
    if rank < 0 or n_per_rank < 1:
        raise ValueError("rank must be >= 0 and n_per_rank >= 1")
    base = rank * n_per_rank
    if base + n_per_rank > 1 << 32:
        raise ValueError("global env ids exceed 2^32")
    return base, n_per_rank


def max_over_ranks(value: float, dist=None, device=None) -> float:
    """The largest value over all ranks (the slowest rank's time)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist=None):
    if dist is not None and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


def mean_over_ranks(vec, dist=None):
    """Average a tensor over all ranks in place (sum all-reduce, then divide):
    the gradient exchange of a data-parallel update.  Returns vec."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return vec
    dist.all_reduce(vec, op=dist.ReduceOp.SUM)
    vec.div_(dist.get_world_size())
    return vec
