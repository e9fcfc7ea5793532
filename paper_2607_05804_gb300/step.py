"""One TurnOPD loss step on the GPU through the C ABI: blend weights, loss +
student-logit gradient, turn statistics.  Buffers come from torch (device
memory only); every computation is a libturnopd kernel.
"""
from __future__ import annotations

import torch

from . import (TURNOPD_FULL_VOCAB, TURNOPD_SCOPE_TRAJ, turnopd_loss_fwd_bwd,
               turnopd_loss_workspace_bytes, turnopd_topk_loss_fwd_bwd, turnopd_turn_counts,
               turnopd_turn_stats, turnopd_weights, turnopd_weights_workspace_bytes)


class LossStep:
    """Holds the per-batch metadata and output buffers of one packed batch.

    turn_id int32[T], loss_mask uint8[T], traj_offsets int64[B+1] (device),
    row_of_token int32[T] or None, sampled_ids int32[T] or None.  k_top > 0 selects the
    teacher top-K reverse KL (sparse outputs topk_ids / topk_grad [T, k_top]).
    """

    def __init__(self, turn_id, loss_mask, traj_offsets, max_turns, vocab, *, row_of_token=None,
                 sampled_ids=None, mode=TURNOPD_FULL_VOCAB, alpha=0.5, scope=TURNOPD_SCOPE_TRAJ,
                 n_min=0, flags=0, k_top=0, device=None):
        dev = turn_id.device if device is None else torch.device(device)
        self.turn_id, self.loss_mask, self.traj_offsets = turn_id, loss_mask, traj_offsets
        self.row_of_token, self.sampled_ids = row_of_token, sampled_ids
        self.max_turns, self.vocab = int(max_turns), int(vocab)
        self.mode, self.alpha, self.scope, self.n_min, self.flags = mode, alpha, scope, n_min, flags
        T, B = turn_id.numel(), traj_offsets.numel() - 1
        self.T, self.B = T, B
        u8 = dict(dtype=torch.uint8, device=dev)
        self.ws_w = torch.empty(max(turnopd_weights_workspace_bytes(B, max_turns), 256), **u8)
        self.ws_l = torch.empty(max(turnopd_loss_workspace_bytes(T), 256), **u8)
        self.w = torch.zeros(max(T, 1), dtype=torch.float32, device=dev)
        self.token_loss = torch.zeros(max(T, 1), dtype=torch.float32, device=dev)
        self.loss = torch.zeros(1, dtype=torch.float64, device=dev)
        self.traj_turn_sum = torch.zeros(max(B * max_turns, 1), dtype=torch.float64, device=dev)
        self.traj_turn_cnt = torch.zeros(max(B * max_turns, 1), dtype=torch.int32, device=dev)
        self.turn_sum = torch.zeros(max_turns, dtype=torch.float64, device=dev)
        self.turn_cnt = torch.zeros(max_turns, dtype=torch.int64, device=dev)
        self.turn_surv = torch.zeros(max_turns, dtype=torch.int32, device=dev)
        self.counts = torch.zeros(2 * max_turns + 1, dtype=torch.int64, device=dev)
        self.dev_status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.k_top = int(k_top)
        if self.k_top > 0:
            self.topk_ids = torch.full((max(T, 1), self.k_top), -1, dtype=torch.int32, device=dev)
            self.topk_grad = torch.zeros((max(T, 1), self.k_top), dtype=torch.float32, device=dev)

    def local_counts(self, stream=None):
        """Per-rank count vector (sum it over data-parallel ranks for global_counts)."""
        turnopd_turn_counts(self.turn_id, self.loss_mask, self.traj_offsets, self.max_turns,
                            self.traj_turn_cnt, self.counts, self.dev_status, stream)
        return self.counts

    def weights(self, global_counts=None, stream=None):
        turnopd_weights(self.turn_id, self.loss_mask, self.traj_offsets, self.max_turns,
                        self.alpha, self.scope, self.n_min, global_counts, self.w[:self.T],
                        self.ws_w, self.dev_status, stream)
        return self.w[:self.T]

    def loss_fwd_bwd(self, z_student, z_teacher, grad=None, stream=None):
        if self.k_top > 0:
            turnopd_topk_loss_fwd_bwd(z_student, z_teacher, self.vocab, self.row_of_token,
                                      self.loss_mask, self.w[:self.T], self.k_top,
                                      self.topk_ids[:self.T], self.topk_grad[:self.T], grad,
                                      self.flags, self.token_loss[:self.T], self.loss, self.ws_l,
                                      self.dev_status, stream)
            return self.loss
        turnopd_loss_fwd_bwd(z_student, z_teacher, self.vocab, self.row_of_token, self.sampled_ids,
                             self.loss_mask, self.w[:self.T], self.mode, grad, self.flags,
                             self.token_loss[:self.T], self.loss, self.ws_l, self.dev_status,
                             stream)
        return self.loss

    def turn_stats(self, stream=None):
        turnopd_turn_stats(self.token_loss[:self.T], self.turn_id, self.loss_mask,
                           self.traj_offsets, self.max_turns, self.traj_turn_sum,
                           self.traj_turn_cnt, self.turn_sum, self.turn_cnt, self.turn_surv,
                           self.dev_status, stream)

    def run(self, z_student, z_teacher, grad=None, global_counts=None, stream=None):
        """The whole hot path: weights -> loss + gradient -> turn statistics."""
        self.weights(global_counts, stream)
        self.loss_fwd_bwd(z_student, z_teacher, grad, stream)
        self.turn_stats(stream)
        return self.loss

    def status(self) -> int:
        return int(self.dev_status.item())

    def stats(self):
        Tm, B = self.max_turns, self.B
        return dict(traj_turn_sum=self.traj_turn_sum[:B * Tm].view(B, Tm),
                    traj_turn_cnt=self.traj_turn_cnt[:B * Tm].view(B, Tm),
                    turn_sum=self.turn_sum, turn_cnt=self.turn_cnt, turn_surv=self.turn_surv)


def to_device(batch, device, compact: bool):
    """Device tensors of a workloads.Batch: (turn_id, loss_mask, traj_offsets, row_of_token)."""
    tid = torch.from_numpy(batch.turn_id).to(device)
    msk = torch.from_numpy(batch.loss_mask).to(device)
    off = torch.from_numpy(batch.traj_offsets).to(device)
    rot = torch.from_numpy(batch.compact_rows()).to(device) if compact else None
    return tid, msk, off, rot
