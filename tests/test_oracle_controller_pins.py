"""Pins of the controller oracle (rollout-depth budgeting, Sec. 4.1 and
Algorithm 1) against closed forms and the properties the paper states."""
import math

import numpy as np
import pytest

from oracle import controller as C


def test_efficiency_is_scale_invariant_and_ignores_negative_kl():
    K = np.array([0.9, 0.4, -0.05, 0.3, 0.2])
    n = np.array([64, 40, 30, 20, 9])
    _, q1, h1, e1 = C.efficiency(K, n)
    _, q2, h2, e2 = C.efficiency(K * 37.0, n)
    np.testing.assert_allclose(q1, q2, rtol=1e-7)
    assert e1 == e2
    m, _, _, _ = C.efficiency(K, n)
    assert m[2] == 0.0


def test_efficiency_closed_forms():
    # all mass at one turn: the centroid is that turn
    K = np.zeros(9); K[6] = 0.5
    assert C.efficiency(K, np.full(9, 10))[3] == 6
    # equal KL: the centroid is the survivor-weighted mean turn index
    n = np.array([8, 4, 2, 1])
    hbar = C.efficiency(np.ones(4), n)[2]
    assert abs(hbar - (0 * 8 + 1 * 4 + 2 * 2 + 3 * 1) / 15) < 1e-8
    # two equal masses at turns 2 and 5: centroid 3.5, rounded half to even -> 4
    # (eps = 0; the paper's eps in q pulls an exact half just below it)
    K = np.zeros(8); K[2] = K[5] = 1.0
    _, _, hbar, he = C.efficiency(K, np.full(8, 3), eps=0.0)
    assert hbar == 3.5 and he == 4
    assert C.efficiency(K, np.full(8, 3))[3] == 3


def test_coverage_quantile_closed_forms():
    assert C.coverage([7] * 12, [True] * 12) == 7
    lens = np.arange(1, 11)
    assert C.coverage(lens, np.ones(10, bool), p=0.8, min_cov_traj=8) == 8
    assert C.coverage(lens, np.ones(10, bool), p=0.5, min_cov_traj=8) == 5
    # fewer than min_cov_traj successes: the previous bound stays
    assert C.coverage(lens, np.arange(10) < 5, min_cov_traj=8, prev=13) == 13
    # use_success off: every probe trajectory counts
    succ = np.arange(10) < 5                       # successes are the short ones (lengths 1..5)
    assert C.coverage(lens, succ, p=0.8, min_cov_traj=5) == 4
    assert C.coverage(lens, succ, p=0.8, min_cov_traj=5, use_success=False) == 8


def test_schedule_and_the_plus_one():
    c = C.Controller(h_min=2, h_max=50, warmup=3, interval=8)
    hhat, probe, roll = c.plan(1)
    assert hhat == 50 and probe and roll == 50       # Hbar_0 = H_max
    assert [k for k in range(1, 40) if C.is_probe(k, 3, 8)] == [1, 2, 3, 8, 16, 24, 32]
    assert C.rollout_depth(4.0, 2, 50) == 5           # 0-based turn index -> depth
    assert C.rollout_depth(0.2, 2, 50) == 2           # clipped at H_min
    assert C.rollout_depth(70.0, 2, 50) == 50


def test_ema_geometric_closed_form():
    a, H0, c_ = 0.3, 50.0, 6
    ctl = C.Controller(h_min=2, h_max=50, ema_alpha=a, warmup=100, interval=8, min_cov_traj=1000)
    K = np.zeros(12); K[c_] = 1.0
    n = np.full(12, 10)
    for j in range(1, 11):
        h = ctl.update(j, K * n, n, n, [], [])
        assert abs(h - (c_ + (H0 - c_) * (1 - a) ** j)) < 1e-9
    # non-probe steps leave the average alone
    ctl2 = C.Controller(warmup=0, interval=8)
    assert ctl2.update(5, K * n, n, n, [], []) == 50.0


def test_controller_takes_the_larger_arm():
    ctl = C.Controller(h_min=2, h_max=50, ema_alpha=1.0, warmup=10, min_cov_traj=4)
    K = np.zeros(10); K[1] = 1.0
    n = np.full(10, 10)
    ctl.update(1, K * n, n, n, [9, 9, 9, 9], [True] * 4)
    assert ctl.h_eff == 1 and ctl.h_cov == 9 and ctl.h_ctrl == 9 and ctl.hbar == 9.0
    assert ctl.plan(2)[0] == 10


def test_diagnostics_shares_and_deep_third():
    s = np.array([6.0, 3.0, 2.0, 1.0, 0.6, 0.4, 0.0])
    cnt = np.array([60, 30, 20, 20, 12, 8, 0])
    surv = np.array([10, 10, 8, 6, 4, 2, 0])
    d = C.diagnostics(s, cnt, surv, n_min=1)
    assert abs(d["b"].sum() - 1) < 1e-12 and abs(d["s"].sum() - 1) < 1e-12
    assert d["prefix"] == 6
    K = s[:6] / cnt[:6]
    assert abs(d["ratio"] - (K[4] + K[5]) / (K[0] + K[1])) < 1e-12
    assert abs(d["support"] - (4 + 2) / 2 / 10) < 1e-12
    assert abs(d["budget"] - (0.6 + 0.4) / 13.0) < 1e-12
    d2 = C.diagnostics(s, cnt, surv, n_min=5)      # reliable prefix: turns 0..3
    assert d2["prefix"] == 4 and abs(d2["support"] - 0.6) < 1e-12
