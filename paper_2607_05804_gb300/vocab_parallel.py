"""Vocabulary-parallel loss step: each rank holds a column shard of the
student and teacher logits; one all-gather of 24 B per supervised token
(the shards' partial row statistics) is the only exchange.  The arithmetic is
in libturnopd; torch.distributed carries the partials (any backend)."""
from __future__ import annotations

import torch

from . import (turnopd_loss_workspace_bytes, turnopd_vocab_shard_loss_grad, turnopd_vocab_shard_stats,
               turnopd_vocab_stats_merge)


def vocab_parallel_loss(z_student, z_teacher, row_of_token, loss_mask, w, grad_shard=None, flags=0,
                        group=None, dev_status=None):
    """This rank's shard [num_rows, shard_vocab] -> (token_loss [T], loss [1] float64).
    grad_shard (optional) receives this rank's gradient columns.  With no process
    group (or a world of one) the shard is the whole vocabulary."""
    import torch.distributed as dist

    dev = z_student.device
    T = loss_mask.numel()
    st = dev_status if dev_status is not None else torch.zeros(1, dtype=torch.int32, device=dev)
    part = torch.empty((max(T, 1), 6), dtype=torch.float32, device=dev)
    ws = torch.empty(max(turnopd_loss_workspace_bytes(T), 256), dtype=torch.uint8, device=dev)
    turnopd_vocab_shard_stats(z_student, z_teacher, row_of_token, loss_mask, part[:T], ws, st)
    world = dist.get_world_size(group) if dist.is_available() and dist.is_initialized() else 1
    if world > 1:
        parts = [torch.empty_like(part) for _ in range(world)]
        dist.all_gather(parts, part, group=group)
        parts = torch.stack(parts)
    else:
        parts = part.unsqueeze(0)
    merged = torch.empty_like(part)
    turnopd_vocab_stats_merge(parts[:, :T].contiguous(), loss_mask, merged[:T])
    token_loss = torch.empty(max(T, 1), dtype=torch.float32, device=dev)
    loss = torch.zeros(1, dtype=torch.float64, device=dev)
    turnopd_vocab_shard_loss_grad(z_student, z_teacher, row_of_token, loss_mask, w, merged[:T], grad_shard, flags,
                                  token_loss[:T], loss, ws, st)
    return token_loss[:T], loss
