"""The library's rollout-depth controller and diagnostics (host C++) against
the controller oracle, on random turn tables and trajectory lengths.  No GPU:
these are host functions of libturnopd."""
import math

import numpy as np
import pytest

from oracle import controller as C


@pytest.fixture(scope="module")
def P():
    from paper_2607_05804_gb300 import build as B

    B.build()
    import paper_2607_05804_gb300 as P

    P.load()
    return P


def random_tables(rng, T):
    cnt = rng.integers(0, 400, T).astype(np.int64)
    cnt[0] = max(cnt[0], 1)
    surv = np.sort(rng.integers(0, 64, T))[::-1].astype(np.int32)
    kl = rng.normal(0.3, 0.4, T)
    s = kl * cnt
    return s, cnt, surv


def near_half(x):
    return abs(x - math.floor(x) - 0.5) < 1e-9


def test_efficiency_matches_oracle(P):
    rng = np.random.default_rng(0)
    for trial in range(200):
        T = int(rng.integers(1, 60))
        s, cnt, surv = random_tables(rng, T)
        m, q, hb, he = P.turnopd_depth_efficiency(s, cnt, surv)
        K = C.turn_kl(s, cnt)
        mr, qr, hbr, her = C.efficiency(K, surv)
        np.testing.assert_array_equal(m, mr)
        np.testing.assert_array_equal(q, qr)
        assert hb == hbr
        if not near_half(hbr):
            assert he == her


def test_coverage_matches_oracle(P):
    rng = np.random.default_rng(1)
    for trial in range(300):
        B = int(rng.integers(0, 80))
        L = rng.integers(0, 60, B)
        succ = rng.random(B) < rng.random()
        p = float(rng.choice([0.5, 0.8, 0.95, 1.0]))
        mc = int(rng.integers(0, 12))
        us = bool(rng.integers(0, 2))
        prev = int(rng.integers(0, 20))
        got = P.turnopd_depth_coverage(L, succ, p, mc, us, prev)
        assert got == C.coverage(L, succ, p, mc, us, prev)


def test_controller_run_matches_oracle(P):
    from paper_2607_05804_gb300.controller import DepthController

    rng = np.random.default_rng(2)
    for h_min, h_max, a, warm, every in [(2, 50, 0.3, 3, 8), (1, 30, 0.5, 0, 4), (3, 12, 1.0, 5, 0)]:
        ctl = DepthController(h_min=h_min, h_max=h_max, ema_alpha=a, warmup_steps=warm, probe_interval=every,
                              min_cov_traj=4)
        ref = C.Controller(h_min=h_min, h_max=h_max, ema_alpha=a, warmup=warm, interval=every, min_cov_traj=4)
        for k in range(1, 41):
            assert ctl.plan(k) == ref.plan(k)
            T = int(rng.integers(1, h_max + 1))
            s, cnt, surv = random_tables(rng, T)
            B = 32
            L = rng.integers(1, h_max + 1, B)
            succ = rng.random(B) < 0.4
            P.turnopd_depth_update(ctl.params, ctl.state, k, s, cnt, surv, L, succ)
            ref.update(k, s, cnt, surv, L, succ)
            assert ctl.state.h_bar == ref.hbar
            assert (ctl.state.h_eff, ctl.state.h_cov, ctl.state.h_ctrl) == (ref.h_eff, ref.h_cov, ref.h_ctrl)


def test_diagnostics_match_oracle(P):
    rng = np.random.default_rng(3)
    for trial in range(100):
        T = int(rng.integers(1, 40))
        s, cnt, surv = random_tables(rng, T)
        n_min = int(rng.integers(0, 20))
        b, sh, deep = P.turnopd_turn_diagnostics(s, cnt, surv, n_min)
        d = C.diagnostics(s, cnt, surv, n_min)
        np.testing.assert_allclose(b, d["b"], rtol=1e-14, atol=0)
        np.testing.assert_allclose(sh, d["s"], rtol=1e-12, atol=1e-15)
        assert deep[0] == d["prefix"]
        for i, key in ((1, "ratio"), (2, "support"), (3, "budget")):
            if math.isnan(d[key]):
                assert math.isnan(deep[i])
            else:
                assert abs(deep[i] - d[key]) <= 1e-12 * max(1.0, abs(d[key]))


def test_errors(P):
    import ctypes

    lib = P.load()
    pr = P.turnopd_depth_default_params()
    st = P.turnopd_depth_init(pr)
    assert lib.turnopd_depth_init(None, ctypes.byref(st)) == 1
    bad = P.turnopd_depth_default_params()
    bad.h_max = 1
    with pytest.raises(P.TurnopdError) as e:
        P.turnopd_depth_init(bad)
    assert e.value.code == 2
    with pytest.raises(P.TurnopdError) as e:
        P.turnopd_depth_plan(pr, st, 0)
    assert e.value.code == 2
    bad = P.turnopd_depth_default_params()
    bad.coverage_p = 1.5
    with pytest.raises(P.TurnopdError):
        P.turnopd_depth_plan(bad, st, 1)
    with pytest.raises(P.TurnopdError) as e:
        P.turnopd_depth_coverage([1, 2], [1, 1], p=0.0)
    assert e.value.code == 2
