"""Rollout-depth controller of TurnOPD (Sec. 4.1, Algorithm 1) on top of a
LossStep: the library's host functions fed with the step's per-turn tables.
"""
from __future__ import annotations

from . import (turnopd_depth_default_params, turnopd_depth_init, turnopd_depth_plan,
               turnopd_depth_update, turnopd_turn_diagnostics)


class DepthController:
    """plan(k) -> (h_hat, is_probe, h_roll) before step k's rollouts;
    update(k, step, traj_len, traj_success) after it (probe steps only change
    the state).  Keyword arguments override turnopd_depth_params fields."""

    def __init__(self, **overrides):
        self.params = turnopd_depth_default_params()
        for k, v in overrides.items():
            if not hasattr(self.params, k):
                raise AttributeError(f"turnopd_depth_params has no field {k}")
            setattr(self.params, k, v)
        self.state = turnopd_depth_init(self.params)

    def plan(self, k: int):
        return turnopd_depth_plan(self.params, self.state, k)

    def update(self, k: int, step, traj_len, traj_success):
        """`step`: a LossStep whose turn_stats() ran on the probe batch."""
        turnopd_depth_update(self.params, self.state, k, step.turn_sum, step.turn_cnt, step.turn_surv,
                             traj_len, traj_success)
        return self.state.h_bar

    @staticmethod
    def diagnostics(step, n_min: int = 1):
        return turnopd_turn_diagnostics(step.turn_sum, step.turn_cnt, step.turn_surv, n_min)
