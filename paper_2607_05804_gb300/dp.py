"""Data-parallel host logic: ranks hold whole trajectories.

The only data the loss path exchanges across ranks is
  * before the weights: the count vector [S_t, C_t, B'] of turnopd_turn_counts
    (2 * max_turns + 1 int64 values), summed over ranks and passed to
    turnopd_weights as `global_counts`;
  * after the step: the weighted loss and the turn statistics, all sums.
Each is one sum all-reduce of a few hundred numbers through torch.distributed.
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
    (per-trajectory tables stay with the rank that owns the trajectory), in ONE
    all-reduce: the four tensors travel packed in a float64 buffer
    [loss, turn_sum, turn_cnt, turn_surv].  The counts ride as doubles, which hold
    every integer below 2^53 exactly, far above any token count a step can have,
    so they come back bit-exact."""
    import torch
    import torch.distributed as dist

    if dist.is_initialized() and dist.get_world_size(group) > 1:
        parts = (loss, turn_sum, turn_cnt, turn_surv)
        sizes = [t.numel() for t in parts]
        buf = torch.cat([t.reshape(-1).to(torch.float64) for t in parts])
        dist.all_reduce(buf, op=dist.ReduceOp.SUM, group=group)
        for t, piece in zip(parts, torch.split(buf, sizes)):
            t.copy_(piece.reshape(t.shape).to(t.dtype))
    return loss, turn_sum, turn_cnt, turn_surv
