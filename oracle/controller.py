"""Reference (oracle) for TurnOPD's adaptive rollout-depth controller and the
turn-level loss-allocation diagnostics.

TEST INFRASTRUCTURE ONLY: nothing on the product path imports this module.
Plain Python/numpy, float64, written from the paper's definitions:

  efficiency mass   m_t = [K_t]_+ n_t / n_0,  q_t = m_t / (sum_j m_j + eps),
                    Hbar_eff = sum_t t q_t,  H_eff = round(Hbar_eff)
                    (Sec. 4.1, "Efficiency-side Mass"; t is the 0-based turn index)
  coverage bound    F(H) = 1 - n_{H+1} / n_1 over the successful probe
                    trajectories (all trajectories when use_success is off),
                    H_cov = min{H : F(H) >= p}, refreshed only when at least
                    min_cov_traj successful trajectories were probed
                    (Sec. 4.1, "Coverage-side Lower Bound"; full configuration
                    table: coverage_quantile, use_success, min_cov_traj)
  update            H_ctrl = max(H_eff, H_cov);  Hbar_k = (1 - a) Hbar_{k-1} + a H_ctrl
                    on probe steps, Hbar_k = Hbar_{k-1} otherwise
                    (Sec. 4.1, "Dynamic Update"; Algorithm 1)
  schedule          Hhat_k = clip(round(Hbar_{k-1}) + 1, H_min, H_max);
                    probe_k = (k <= K_warm) or (k mod r_probe == 0);
                    H_roll = H_max on probe steps, Hhat_k otherwise;
                    Hbar_0 = H_max, H_cov = 0 at the start (Algorithm 1)
  diagnostics       b_t = n_t / N (token share), s_t = sum_i l_{t,i} / sum l
                    (loss share) (Sec. 3, "Loss-allocation diagnostics"), and the
                    deep-third figures of the loss-allocation table.

round() is round-half-to-even (Python's round and C's nearbyint under the
default rounding mode agree on it).
"""
from __future__ import annotations

import math

import numpy as np


def turn_kl(turn_sum, turn_cnt):
    """K_t = pooled per-token KL at turn index t (0 where no token)."""
    s = np.asarray(turn_sum, np.float64)
    c = np.asarray(turn_cnt, np.float64)
    return np.where(c > 0, s / np.where(c > 0, c, 1.0), 0.0)


def efficiency(K, n, eps=1e-8):
    """-> (m, q, Hbar_eff, H_eff) from K_t and survivor counts n_t (n_0 = n[0])."""
    K = np.asarray(K, np.float64)
    n = np.asarray(n, np.float64)
    T = K.size
    m = np.zeros(T)
    if T and n[0] > 0:
        for t in range(T):
            m[t] = max(K[t], 0.0) * n[t] / n[0]
    total = 0.0
    for t in range(T):
        total += m[t]
    q = m / (total + eps)
    hbar = 0.0
    for t in range(T):
        hbar += t * q[t]
    return m, q, hbar, int(round(hbar))


def coverage(traj_len, success, p=0.8, min_cov_traj=8, use_success=True, prev=0):
    """H_cov from probe trajectory lengths (turns) and success flags; `prev` is kept
    when fewer than min_cov_traj successful trajectories are available."""
    L = np.asarray(traj_len, np.int64)
    s = np.asarray(success, bool)
    if int(s.sum()) < min_cov_traj:
        return prev
    pool = L[s] if use_success else L
    n1 = int((pool >= 1).sum())
    if n1 == 0:
        return prev
    H = 0
    while True:
        n_next = int((pool >= H + 1).sum())   # trajectories that reach turn H + 1
        if 1.0 - n_next / n1 >= p:
            return H
        H += 1


def rollout_depth(hbar_prev, h_min, h_max):
    return min(max(int(round(hbar_prev)) + 1, h_min), h_max)


def is_probe(k, warmup, interval):
    return k <= warmup or (interval > 0 and k % interval == 0)


class Controller:
    """The controller state machine of Algorithm 1."""

    def __init__(self, h_min=2, h_max=50, ema_alpha=0.30, p=0.80, min_cov_traj=8, use_success=True,
                 warmup=3, interval=8, eps=1e-8):
        self.h_min, self.h_max, self.a, self.p = h_min, h_max, ema_alpha, p
        self.min_cov, self.use_success, self.warmup, self.interval, self.eps = (
            min_cov_traj, use_success, warmup, interval, eps)
        self.hbar = float(h_max)
        self.h_cov = 0
        self.h_eff = 0
        self.h_ctrl = 0

    def plan(self, k):
        """Step k (1-based): (Hhat_k, probe_k, H_roll)."""
        hhat = rollout_depth(self.hbar, self.h_min, self.h_max)
        probe = is_probe(k, self.warmup, self.interval)
        return hhat, probe, (self.h_max if probe else hhat)

    def update(self, k, turn_sum, turn_cnt, turn_surv, traj_len, success):
        """After step k: a probe step refreshes H_eff, H_cov and the EMA."""
        if not is_probe(k, self.warmup, self.interval):
            return self.hbar
        K = turn_kl(turn_sum, turn_cnt)
        _, _, _, self.h_eff = efficiency(K, turn_surv, self.eps)
        self.h_cov = coverage(traj_len, success, self.p, self.min_cov, self.use_success, self.h_cov)
        self.h_ctrl = max(self.h_eff, self.h_cov)
        self.hbar = (1.0 - self.a) * self.hbar + self.a * self.h_ctrl
        return self.hbar


def diagnostics(turn_sum, turn_cnt, turn_surv, n_min=1):
    """Per turn index: b_t = n_t / N, s_t = sum l / total; and over the reliable
    prefix (turns 0.. while turn_surv >= n_min), with third = floor(P / 3) turns
    at each end: deep/shallow ratio of mean K_t, deep support = mean n_t / n_0
    over the deep third, deep loss budget = sum of s_t over the deep third.
    -> dict (the deep figures are nan when the prefix is shorter than 3)."""
    s = np.asarray(turn_sum, np.float64)
    c = np.asarray(turn_cnt, np.float64)
    n = np.asarray(turn_surv, np.float64)
    N = c.sum()
    Ls = s.sum()
    b = c / N if N > 0 else np.zeros_like(c)
    sh = s / Ls if Ls != 0 else np.zeros_like(s)
    P = 0
    while P < n.size and n[P] >= n_min and n[P] > 0:
        P += 1
    out = dict(b=b, s=sh, prefix=P, ratio=math.nan, support=math.nan, budget=math.nan)
    third = P // 3
    if third >= 1:
        K = turn_kl(s, c)
        shallow = range(0, third)
        deep = range(P - third, P)
        ks = sum(K[t] for t in shallow) / third
        kd = sum(K[t] for t in deep) / third
        out["ratio"] = kd / ks if ks != 0 else math.nan
        out["support"] = sum(n[t] for t in deep) / third / n[0]
        out["budget"] = sum(sh[t] for t in deep)
    return out
