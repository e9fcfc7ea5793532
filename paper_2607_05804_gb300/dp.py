"""Data-parallel host logic: ranks hold whole trajectories.

The only data the loss path exchanges across ranks is
  * before the weights: the count vector [S_t, C_t, B'] of turnopd_turn_counts
    (2 * max_turns + 1 int64 values), summed over ranks and passed to
    turnopd_weights as `global_counts`;
  * after the step: the weighted loss and the turn statistics, all sums.
Both are sum all-reduces of a few hundred numbers through torch.distributed.
"""
from __future__ import annotations


def global_counts(local_counts, group=None):
    """Sum of every rank's count vector (a new tensor; the input is left as is)."""
    import torch.distributed as dist

    out = local_counts.clone()
    if dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(out, op=dist.ReduceOp.SUM, group=group)
    return out


def reduce_step(loss, turn_sum, turn_cnt, turn_surv, group=None):
    """In-place sums over ranks of the batch loss and the per-turn-index statistics
    (per-trajectory tables stay with the rank that owns the trajectory)."""
    import torch.distributed as dist

    if dist.is_initialized() and dist.get_world_size(group) > 1:
        for t in (loss, turn_sum, turn_cnt, turn_surv):
            dist.all_reduce(t, op=dist.ReduceOp.SUM, group=group)
    return loss, turn_sum, turn_cnt, turn_surv
