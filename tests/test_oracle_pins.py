"""Pins for the fp64 CPU oracle: each test ties it to something other than
itself -- hand-worked values, closed forms, textbook/library routines,
invariants the mathematics fixes, finite differences and brute force.

TurnOPD (arXiv 2607.05804) passages pinned: Eq. (opd-rkl) (per-token reverse
KL and its gradient), Sec. 5.2 and Algorithm 1 (blend weights and the alpha
schedule), Eq. (observed-turn-kl) and Sec. 5.1 (turn statistics), Prop. 1 and
its proof (joint convexity, KL(p||p) = 0), the KL-normaliser ablation table
(printed alpha per training phase), the hyper-parameter table (n_min floor).
"""
from fractions import Fraction
import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats

import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------- helpers

def brute_counts(b: W.Batch):
    """Direct Python loops over every token (independent of the oracle)."""
    B, Tm = b.num_traj, b.max_turns
    n = [[0] * Tm for _ in range(B)]
    for bb in range(B):
        for i in range(int(b.traj_offsets[bb]), int(b.traj_offsets[bb + 1])):
            if b.loss_mask[i]:
                n[bb][int(b.turn_id[i])] += 1
    S = [sum(1 for bb in range(B) if n[bb][t] > 0) for t in range(Tm)]
    C = [sum(n[bb][t] for bb in range(B)) for t in range(Tm)]
    Bp = sum(1 for bb in range(B) if sum(n[bb]) > 0)
    return np.array(n, np.int32).reshape(B, Tm), np.array(S + C + [Bp], np.int64)


def random_batches(seed, count=6):
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(count):
        out.append(W.random_structure(rng, num_traj=int(rng.integers(1, 7)),
                                      max_len=int(rng.integers(1, 60)),
                                      max_turns=int(rng.integers(1, 9))))
    return out


def f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


# ----------------------------------------------------------------- metadata

def test_counts_match_brute_force(oracle):
    for b in random_batches(1, 20) + [W.tiny(), W.packed(3), W.household(2)]:
        n_bt, counts = oracle.turn_counts(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        n_ref, c_ref = brute_counts(b)
        assert np.array_equal(n_bt, n_ref)
        assert np.array_equal(counts, c_ref)
        Tm = b.max_turns
        assert counts[Tm:2 * Tm].sum() == b.loss_mask.sum()
        assert counts[:Tm].sum() == (n_ref > 0).sum()


def test_counts_errors(oracle):
    b = W.tiny()
    tid = b.turn_id.copy()
    tid[20] = 7  # supervised token (second assistant span of traj 0) with turn 7 >= 4
    assert b.loss_mask[20] == 1
    with pytest.raises(oracle.OracleError) as e:
        oracle.turn_counts(tid, b.loss_mask, b.traj_offsets, b.max_turns)
    assert e.value.code == 4
    tid = b.turn_id.copy()
    tid[0] = 99  # masked token: its turn id is ignored
    oracle.turn_counts(tid, b.loss_mask, b.traj_offsets, b.max_turns)
    off = b.traj_offsets.copy()
    off[1] = off[2] + 1  # non-monotone
    with pytest.raises(oracle.OracleError) as e:
        oracle.turn_counts(b.turn_id, b.loss_mask, off, b.max_turns)
    assert e.value.code == 3


# ----------------------------------------------------------------- weights

def parse_golden_weights():
    cases, ex = [], None
    with open(os.path.join(GOLDEN, "weights_worked_examples.txt")) as fh:
        for line in fh:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, _, val = line.partition(":")
            val = val.strip()
            if key == "example":
                ex = dict(name=val, trajs=[], max_turns=None)
            elif key == "max_turns":
                ex["max_turns"] = int(val)
            elif key == "traj":
                ex["trajs"].append(val.split())
            elif key == "case":
                kv = dict(x.split("=") for x in val.split())
                cur = dict(example=ex, scope=kv["scope"], alpha=float(kv["alpha"]),
                           n_min=int(kv["n_min"]))
                cases.append(cur)
            elif key == "w":
                cur["w"] = [Fraction(x) for x in val.split()]
    return cases


def golden_batch(ex):
    tid, msk, off = [], [], [0]
    for toks in ex["trajs"]:
        for t in toks:
            if t == "o":
                tid.append(-1)
                msk.append(0)
            else:
                tid.append(int(t))
                msk.append(1)
        off.append(off[-1] + len(toks))
    return (np.array(tid, np.int32), np.array(msk, np.uint8), np.array(off, np.int64),
            ex["max_turns"])


@pytest.mark.parametrize("case", parse_golden_weights(),
                         ids=lambda c: f"{c['example']['name']}-{c['scope']}-a{c['alpha']}-n{c['n_min']}")
def test_weights_hand_worked(oracle, case):
    tid, msk, off, Tm = golden_batch(case["example"])
    scope = oracle.SCOPE_TRAJ if case["scope"] == "traj" else oracle.SCOPE_BATCH
    w = oracle.weights(tid, msk, off, Tm, case["alpha"], scope, case["n_min"])
    ref = np.array([float(x) for x in case["w"]])
    assert w.shape == ref.shape
    np.testing.assert_allclose(w, ref, rtol=1e-15, atol=0)
    assert sum(case["w"]) == 1


@pytest.mark.parametrize("scope", [0, 1])
def test_weights_invariants(oracle, scope):
    for b in random_batches(7, 25) + [W.packed(1), W.household(1), W.multihop(1)]:
        args = (b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        n_bt, counts = oracle.turn_counts(*args)
        Tm = b.max_turns
        Bp = counts[2 * Tm]
        w0 = oracle.weights(*args, 0.0, scope)
        w1 = oracle.weights(*args, 1.0, scope)
        w3 = oracle.weights(*args, 0.3, scope)
        if Bp == 0:
            assert not w0.any() and not w1.any()
            continue
        # normalisation and linearity in alpha
        for w in (w0, w1, w3):
            assert math.isclose(w.sum(), 1.0, rel_tol=1e-12)
            assert (w[b.loss_mask == 0] == 0).all()
            assert (w[b.loss_mask == 1] > 0).all()
        np.testing.assert_allclose(w3, 0.7 * w0 + 0.3 * w1, rtol=1e-13)
        off = b.traj_offsets
        N = counts[Tm:2 * Tm].sum()
        S = counts[:Tm].sum()
        for bb in range(b.num_traj):
            sl = slice(off[bb], off[bb + 1])
            m = b.loss_mask[sl] == 1
            Nb = int(m.sum())
            if Nb == 0:
                continue
            if scope == 0:
                # alpha = 0: seq-mean-token-mean, 1/(B' N_b) per token
                np.testing.assert_allclose(w0[sl][m], 1.0 / (Bp * Nb), rtol=1e-14)
                assert math.isclose(w1[sl].sum(), 1.0 / Bp, rel_tol=1e-12)
            else:
                np.testing.assert_allclose(w0[sl][m], 1.0 / N, rtol=1e-14)
            # alpha = 1: equal mass per non-empty turn
            tb = b.turn_id[sl][m]
            turns = np.unique(tb)
            for t in turns:
                mass = w1[sl][m][tb == t].sum()
                expect = 1.0 / (Bp * turns.size) if scope == 0 else 1.0 / S
                assert math.isclose(mass, expect, rel_tol=1e-12)


def test_weights_equal_turns_alpha_free(oracle):
    """When every turn of a trajectory has the same token count, token mass and turn
    mass coincide and alpha has no effect (Sec. 5.2: q^traj = q^turn)."""
    spans = [[("o", 3), ("a", 4)] * 3, [("a", 2), ("o", 1), ("a", 2)], [("o", 5)]]
    b = W._from_spans("eq", spans, max_turns=4)
    args = (b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    np.testing.assert_allclose(oracle.weights(*args, 0.0), oracle.weights(*args, 1.0), rtol=1e-15)


def test_weights_floor_disabled_equivalences(oracle):
    for b in random_batches(11, 15):
        args = (b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        for scope in (0, 1):
            ref = oracle.weights(*args, 0.6, scope, 0)
            # every non-empty turn index is reached by >= 1 trajectory
            np.testing.assert_allclose(oracle.weights(*args, 0.6, scope, 1), ref, rtol=1e-15)
            # a floor above the batch size makes every turn unreliable: alpha drops out
            big = b.num_traj + 1
            np.testing.assert_allclose(oracle.weights(*args, 0.6, scope, big),
                                       oracle.weights(*args, 0.0, scope, big), rtol=1e-15)


def test_weights_floor_keeps_token_mass(oracle):
    """Unreliable turns keep exactly their token-level mass U_b/N_b (traj scope)."""
    for b in random_batches(21, 20):
        args = (b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        n_bt, counts = oracle.turn_counts(*args)
        Tm = b.max_turns
        n_min = 2
        S = counts[:Tm]
        Bp = counts[2 * Tm]
        if Bp == 0:
            continue
        w1 = oracle.weights(*args, 1.0, 0, n_min)
        assert math.isclose(w1.sum(), 1.0, rel_tol=1e-12)
        off = b.traj_offsets
        for bb in range(b.num_traj):
            Nb = n_bt[bb].sum()
            if Nb == 0:
                continue
            unrel = [t for t in range(Tm) if S[t] < n_min and n_bt[bb, t] > 0]
            Ub = sum(n_bt[bb, t] for t in unrel)
            sl = slice(off[bb], off[bb + 1])
            m = (b.loss_mask[sl] == 1) & np.isin(b.turn_id[sl], unrel)
            assert math.isclose(w1[sl][m].sum(), Ub / (Nb * Bp), rel_tol=1e-12, abs_tol=1e-300)


def test_weights_global_counts_split(oracle):
    """Data-parallel reading: splitting trajectories over ranks and summing the
    count vectors reproduces the single-batch weights (traj and batch scope, floor on)."""
    rng = np.random.default_rng(5)
    for _ in range(10):
        b = W.random_structure(rng, num_traj=6, max_len=40, max_turns=5, allow_empty=True)
        args = (b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        cut = int(rng.integers(1, 6))
        parts = []
        for lo, hi in ((0, cut), (cut, b.num_traj)):
            a, z = b.traj_offsets[lo], b.traj_offsets[hi]
            parts.append((b.turn_id[a:z], b.loss_mask[a:z], b.traj_offsets[lo:hi + 1] - a))
        g = sum(oracle.turn_counts(*p, b.max_turns)[1] for p in parts)
        for scope in (0, 1):
            for n_min in (0, 2):
                ref = oracle.weights(*args, 0.4, scope, n_min)
                got = np.concatenate([oracle.weights(*p, b.max_turns, 0.4, scope, n_min,
                                                     global_counts=g) for p in parts])
                np.testing.assert_allclose(got, ref, rtol=1e-15, atol=0)


def test_alpha_schedule_matches_printed_phases(oracle):
    """KL-normaliser ablation: alpha per early/mid/late third of K = 100 steps is
    printed as 0.17 / 0.50 / 0.83 with s, e = 0, 1 (hyper-parameter table)."""
    K = 100
    a = [oracle.alpha_schedule(k, K, 0.0, 1.0) for k in range(1, K + 1)]
    thirds = [np.mean(a[0:33]), np.mean(a[33:66]), np.mean(a[66:100])]
    for got, printed in zip(thirds, (0.17, 0.50, 0.83)):
        assert abs(got - printed) <= 0.005 + 1e-12
    assert oracle.alpha_schedule(0, K) == 0.0 and oracle.alpha_schedule(K, K) == 1.0
    assert oracle.alpha_schedule(10, 100, 0.2, 0.6) == 0.0
    assert oracle.alpha_schedule(90, 100, 0.2, 0.6) == 1.0
    assert math.isclose(oracle.alpha_schedule(40, 100, 0.2, 0.6), 0.5, rel_tol=1e-15)


# ----------------------------------------------------------------- KL value

def kl_of(oracle, zs, zt, **kw):
    return oracle.row(f32(zs), f32(zt), **kw)


def test_kl_self_is_zero_and_shift_invariant(oracle):
    rng = np.random.default_rng(0)
    dyadic = lambda n: np.round(rng.normal(0, 3, n) * 1024) / 1024  # shifts stay exact in fp32
    for V in (1, 2, 7, 1024):
        z = dyadic(V)
        _, _, kl, _, g = kl_of(oracle, z, z)
        assert abs(kl) < 1e-12 and np.abs(g).max() < 1e-12
        # both rows shifted by different constants: distributions unchanged
        zt = dyadic(V)
        base = kl_of(oracle, z, zt)
        sh = kl_of(oracle, z + 4.0, zt - 2.5)
        assert math.isclose(base[2], sh[2], rel_tol=1e-12, abs_tol=1e-14)
        np.testing.assert_allclose(base[4], sh[4], rtol=1e-9, atol=1e-15)


def test_kl_nonnegative_and_matches_scipy(oracle):
    rng = np.random.default_rng(1)
    for V in (2, 3, 50, 1000):
        for _ in range(5):
            zs = f32(rng.normal(0, 2, V))
            zt = f32(rng.normal(0, 2, V))
            lse_s, lse_t, kl, klf, _ = oracle.row(zs, zt)
            assert kl >= 0 and kl == klf
            ps = scipy.special.softmax(zs.astype(np.float64))
            pt = scipy.special.softmax(zt.astype(np.float64))
            assert math.isclose(kl, scipy.stats.entropy(ps, pt), rel_tol=1e-10, abs_tol=1e-13)
            assert math.isclose(lse_s, scipy.special.logsumexp(zs.astype(np.float64)), rel_tol=1e-14)
            assert math.isclose(lse_t, scipy.special.logsumexp(zt.astype(np.float64)), rel_tol=1e-14)


@pytest.mark.parametrize("V,c", [(2, 1.0), (1024, 8.0), (151936, 8.0), (5, -3.0)])
def test_kl_uniform_vs_spike_closed_forms(oracle, V, c):
    uni = np.zeros(V)
    spike = np.zeros(V)
    spike[V // 3] = c
    # uniform student vs spiked teacher: -log V + log(e^c + V - 1) - c/V
    kl = kl_of(oracle, uni, spike)[2]
    ref = -math.log(V) + math.log(math.exp(c) + V - 1) - c / V
    assert math.isclose(kl, ref, rel_tol=1e-12, abs_tol=1e-13)
    # spiked student vs uniform teacher: log V - H(p_s)
    Z = math.exp(c) + V - 1
    p1, p0 = math.exp(c) / Z, 1.0 / Z
    H = -(p1 * math.log(p1) + (V - 1) * p0 * math.log(p0))
    kl = kl_of(oracle, spike, uni)[2]
    assert math.isclose(kl, math.log(V) - H, rel_tol=1e-11, abs_tol=1e-13)


def test_kl_bernoulli(oracle):
    rng = np.random.default_rng(2)
    for _ in range(20):
        zs, zt = rng.normal(0, 2, 2), rng.normal(0, 2, 2)
        zs, zt = f32(zs).astype(np.float64), f32(zt).astype(np.float64)
        a = 1.0 / (1.0 + math.exp(zs[0] - zs[1]))  # P(student picks 1)
        b = 1.0 / (1.0 + math.exp(zt[0] - zt[1]))
        ref = a * math.log(a / b) + (1 - a) * math.log((1 - a) / (1 - b))
        assert math.isclose(kl_of(oracle, zs, zt)[2], ref, rel_tol=1e-11, abs_tol=1e-14)


def test_kl_permutation_invariance(oracle):
    rng = np.random.default_rng(3)
    V = 300
    zs, zt = f32(rng.normal(0, 3, V)), f32(rng.normal(0, 3, V))
    perm = rng.permutation(V)
    y = 17
    for mode in (0, 1):
        a = oracle.row(zs, zt, mode=mode, y=y, w=0.7)
        b = oracle.row(zs[perm], zt[perm], mode=mode, y=int(np.nonzero(perm == y)[0][0]), w=0.7)
        assert math.isclose(a[2], b[2], rel_tol=1e-12, abs_tol=1e-14)
        np.testing.assert_allclose(a[4][perm], b[4], rtol=1e-11, atol=1e-15)


def test_contamination_compression_bound(oracle):
    """Prop. 1: KL(l pF + (1-l) pS || l pF + (1-l) pT) <= (1-l) KL(pS || pT)."""
    rng = np.random.default_rng(4)
    for _ in range(50):
        V = int(rng.integers(2, 40))
        pF, pS, pT = (rng.dirichlet(np.full(V, 0.5)) for _ in range(3))
        lam = float(rng.random())
        mix_s = lam * pF + (1 - lam) * pS
        mix_t = lam * pF + (1 - lam) * pT
        # rows are logits; use fp32 inputs of log-probabilities
        lhs = kl_of(oracle, np.log(mix_s), np.log(mix_t))[2]
        rhs = (1 - lam) * kl_of(oracle, np.log(pS), np.log(pT))[2]
        assert lhs <= rhs + 1e-6 * (1 + rhs)


# ----------------------------------------------------------------- gradient

def test_grad_finite_differences(oracle):
    """g = w dKL/dz_s by central differences (h = 1e-6) at V <= 16."""
    rng = np.random.default_rng(5)
    for V in (1, 2, 5, 16):
        for _ in range(3):
            # fp32-representable base point; perturbed copies are widened exactly
            zs = f32(rng.normal(0, 2, V)).astype(np.float64)
            zt = f32(rng.normal(0, 2, V)).astype(np.float64)
            w = 0.37
            g = oracle.row(f32(zs), f32(zt), w=w)[4]
            h = 1.0 / 1024  # exactly representable, fp32 steps keep the inputs exact
            for v in range(V):
                e = np.zeros(V)
                e[v] = h
                up = oracle.row(f32(zs + e), f32(zt))[2]
                dn = oracle.row(f32(zs - e), f32(zt))[2]
                fd = w * (up - dn) / (2 * h)
                assert abs(fd - g[v]) <= 2e-6 * (1 + abs(g[v])), (V, v, fd, g[v])


def test_grad_rows_sum_to_zero(oracle):
    rng = np.random.default_rng(6)
    for mode in (0, 1):
        for V in (3, 1024, 151936):
            zs, zt = f32(rng.normal(0, 3, V)), f32(rng.normal(0, 3, V))
            g = oracle.row(zs, zt, mode=mode, y=int(rng.integers(0, V)), w=1.3)[4]
            assert abs(g.sum()) <= 1e-12 * max(1.0, np.abs(g).max() * 10)


def test_sampled_mode_exact_expectation(oracle):
    """E_{y ~ p_s}[l(y)] = KL and E_{y ~ p_s}[g(y)] = g_full, by enumeration over y."""
    rng = np.random.default_rng(7)
    for V in (2, 5, 64):
        zs, zt = f32(rng.normal(0, 2, V)), f32(rng.normal(0, 2, V))
        lse_s, _, kl, _, gfull = oracle.row(zs, zt, mode=0, w=0.9)
        p = np.exp(zs.astype(np.float64) - lse_s)
        el, eg = 0.0, np.zeros(V)
        for y in range(V):
            _, _, l, kl2, g = oracle.row(zs, zt, mode=1, y=y, w=0.9)
            assert kl2 == kl
            el += p[y] * l
            eg += p[y] * g
        assert math.isclose(el, kl, rel_tol=1e-11, abs_tol=1e-14)
        np.testing.assert_allclose(eg, gfull, rtol=1e-9, atol=1e-14)


def test_sampled_gradient_at_a_dominant_token(oracle):
    """Sampled token y whose student logit c stands above V - 1 zeros: p_y = e^c / (e^c + V - 1),
    so g_y = w l (V - 1) / (e^c + V - 1) and g_v = -w l / (e^c + V - 1) in closed form, with
    1 - p_y down to ~6e-13 at c = 40 (where 1 - p_y formed by subtraction keeps only ~4
    digits even in fp64, and none in fp32)."""
    rng = np.random.default_rng(9)
    V = 151936
    for c in (10.0, 20.0, 30.0, 40.0):
        y = int(rng.integers(0, V))
        zs = np.zeros(V, np.float32)
        zs[y] = c
        zt = f32(rng.normal(0, 2, V))
        lse_s, lse_t, l, _, g = oracle.row(zs, zt, mode=1, y=y, w=0.7)
        den = math.exp(c) + (V - 1)
        assert math.isclose(lse_s, math.log(den), rel_tol=1e-14)
        lse_t_ref = float(np.logaddexp.reduce(zt.astype(np.float64)))
        assert math.isclose(l, (c - float(zt[y])) - (math.log(den) - lse_t_ref), rel_tol=1e-12, abs_tol=1e-12)
        assert math.isclose(g[y], 0.7 * l * (V - 1) / den, rel_tol=1e-10)
        others = np.delete(g, y)
        np.testing.assert_allclose(others, -0.7 * l / den, rtol=1e-12)


def test_sampled_mode_monte_carlo(oracle):
    """V = 1024: the sample mean of l(y), y drawn from softmax(z_s), lies within 5 sigma of KL."""
    rng = np.random.default_rng(8)
    V = 1024
    zs, zt = f32(rng.normal(0, 2, V)), f32(rng.normal(0, 2, V))
    lse_s, lse_t, kl, _, _ = oracle.row(zs, zt, mode=0, grad=False)
    p = np.exp(zs.astype(np.float64) - lse_s)
    ys = rng.choice(V, size=4000, p=p / p.sum())
    ls = np.array([oracle.row(zs, zt, mode=1, y=int(y), grad=False)[2] for y in ys])
    assert abs(ls.mean() - kl) <= 5 * ls.std() / math.sqrt(ys.size)


# ----------------------------------------------------------------- batch loss

def _rows_for(b, kind, V, seed, dtype_np=np.float32):
    import torch

    zs, zt = W.make_logits(b.num_tokens, V, kind, torch.float32, seed)
    return zs.numpy(), zt.numpy()


def test_loss_masking_layouts_and_padding(oracle):
    import torch

    b = W.tiny()
    V = 64
    zs, zt = _rows_for(b, "tiny", V, 0)
    w = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, 0.5).astype(np.float32)
    y = W.sample_ids(torch.from_numpy(zs), 0).numpy()
    for mode in (0, 1):
        g, tl, loss = oracle.loss_fwd_bwd(zs, zt, V, b.loss_mask, w, mode=mode, sampled_ids=y)
        assert (tl[b.loss_mask == 0] == 0).all()
        assert not g[b.loss_mask == 0].any()
        # the loss is the weighted sum of per-token losses
        assert math.isclose(loss, float(np.dot(w.astype(np.float64), tl)), rel_tol=1e-13)
        # compact layout: same rows, gathered
        rot = b.compact_rows()
        idx = np.nonzero(b.loss_mask)[0]
        g2, tl2, loss2 = oracle.loss_fwd_bwd(zs[idx], zt[idx], V, b.loss_mask, w, mode=mode,
                                             row_of_token=rot, sampled_ids=y)
        assert loss2 == loss and np.array_equal(tl2, tl)
        assert np.array_equal(g2, g[idx])
        # padded rows (ld > V): padding is never read
        pad = np.full((zs.shape[0], V + 13), 1e30, np.float32)
        padt = pad.copy()
        pad[:, :V], padt[:, :V] = zs, zt
        g3, tl3, loss3 = oracle.loss_fwd_bwd(pad, padt, V, b.loss_mask, w, mode=mode,
                                             sampled_ids=y)
        assert loss3 == loss and np.array_equal(g3, g)


def test_loss_fd_through_batch(oracle):
    """dL/dz_s of the whole batch loss L = sum_i w_i KL_i by central differences."""
    rng = np.random.default_rng(9)
    b = W.random_structure(rng, num_traj=3, max_len=10, max_turns=3, allow_empty=False)
    V = 6
    zs = f32(rng.normal(0, 2, (b.num_tokens, V)))
    zt = f32(rng.normal(0, 2, (b.num_tokens, V)))
    w = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, 0.5).astype(np.float32)
    g, _, _ = oracle.loss_fwd_bwd(zs, zt, V, b.loss_mask, w)
    h = 1.0 / 1024
    for r in range(b.num_tokens):
        for v in range(V):
            up, dn = zs.copy(), zs.copy()
            up[r, v] += h
            dn[r, v] -= h
            fd = (oracle.loss_fwd_bwd(up, zt, V, b.loss_mask, w, grad=False)[2]
                  - oracle.loss_fwd_bwd(dn, zt, V, b.loss_mask, w, grad=False)[2]) / (2 * h)
            assert abs(fd - g[r, v]) <= 2e-6 * (1 + abs(g[r, v]))


def test_loss_errors(oracle):
    b = W.tiny()
    V = 8
    zs = np.zeros((b.num_tokens, V), np.float32)
    w = np.ones(b.num_tokens, np.float32)
    rot = b.compact_rows()
    rot[np.nonzero(b.loss_mask)[0][3]] = -1
    with pytest.raises(oracle.OracleError) as e:
        oracle.loss_fwd_bwd(zs, zs, V, b.loss_mask, w, row_of_token=rot)
    assert e.value.code == 5
    y = np.zeros(b.num_tokens, np.int32)
    y[np.nonzero(b.loss_mask)[0][0]] = V
    with pytest.raises(oracle.OracleError) as e:
        oracle.loss_fwd_bwd(zs, zs, V, b.loss_mask, w, mode=1, sampled_ids=y)
    assert e.value.code == 5
    bad = zs.copy()
    bad[np.nonzero(b.loss_mask)[0][1], 2] = np.inf
    with pytest.raises(oracle.OracleError) as e:
        oracle.loss_fwd_bwd(bad, zs, V, b.loss_mask, w)
    assert e.value.code == 9


def test_bf16_widening_is_exact(oracle):
    """bf16 bit patterns are widened exactly: the bf16 row and its fp32 copy agree bit for bit."""
    import torch

    rng = np.random.default_rng(10)
    x = torch.from_numpy(rng.normal(0, 3, (2, 333)).astype(np.float32)).to(torch.bfloat16)
    bits = W.bf16_bits(x)
    as32 = x.float().numpy()
    a = oracle.row(bits[0], bits[1], w=0.5)
    c = oracle.row(as32[0], as32[1], w=0.5)
    assert a[2] == c[2] and np.array_equal(a[4], c[4])


# ----------------------------------------------------------------- turn stats

def test_turn_stats_brute_force(oracle):
    rng = np.random.default_rng(12)
    for b in random_batches(13, 15) + [W.household(4)]:
        tl = rng.normal(1.0, 0.5, b.num_tokens) * b.loss_mask
        st = oracle.turn_stats(tl, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        n_ref, counts = brute_counts(b)
        Tm = b.max_turns
        assert np.array_equal(st["traj_turn_cnt"], n_ref)
        assert np.array_equal(st["turn_cnt"], counts[Tm:2 * Tm])
        assert np.array_equal(st["turn_surv"], counts[:Tm])
        ref = np.zeros((b.num_traj, Tm))
        for bb in range(b.num_traj):
            for i in range(b.traj_offsets[bb], b.traj_offsets[bb + 1]):
                if b.loss_mask[i]:
                    ref[bb, b.turn_id[i]] += tl[i]
        np.testing.assert_allclose(st["traj_turn_sum"], ref, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(st["turn_sum"], ref.sum(0), rtol=1e-12, atol=1e-12)
        assert math.isclose(st["turn_sum"].sum(), tl.sum(), rel_tol=1e-12, abs_tol=1e-12)


# ----------------------------------------------------------------- fused heads

def test_fused_matches_matmul_then_rows(oracle):
    """z = h W^T by numpy matmul (library primitive), then the pinned row oracle, then
    dh = g W by matmul, against the fused oracle.  Inputs are small dyadic values so
    every logit is exact in fp32 and the row oracle sees the very same logits."""
    import torch

    rng = np.random.default_rng(14)
    T, d_s, d_t, V = 12, 16, 24, 40
    def q(shape, scale):  # multiples of scale/8 in [-scale, scale]: exact in bf16
        return torch.from_numpy(rng.integers(-8, 9, shape).astype(np.float32) * (scale / 8)).to(torch.bfloat16)
    h_s, W_s, h_t, W_t = q((T, d_s), 1.0), q((V, d_s), 0.25), q((T, d_t), 1.0), q((V, d_t), 0.25)
    bits = [W.bf16_bits(x) for x in (h_s, W_s, h_t, W_t)]
    f = [x.double().numpy() for x in (h_s, W_s, h_t, W_t)]
    mask = (rng.random(T) < 0.6).astype(np.uint8)
    w = (rng.random(T) * mask).astype(np.float32)
    y = rng.integers(0, V, T).astype(np.int32)
    zs = f[0] @ f[1].T
    zt = f[2] @ f[3].T
    assert np.array_equal(f32(zs).astype(np.float64), zs) and np.array_equal(f32(zt).astype(np.float64), zt)
    for mode in (0, 1):
        dh, tl, loss, dw = oracle.fused_lmhead(*bits, mask, w, mode=mode, sampled_ids=y, dW=True)
        G = np.zeros((T, V))
        for i in range(T):
            if not mask[i]:
                assert tl[i] == 0 and not dh[i].any()
                continue
            _, _, ell, _, g = oracle.row(f32(zs[i]), f32(zt[i]), mode=mode, y=int(y[i]), w=float(w[i]))
            assert tl[i] == ell
            np.testing.assert_allclose(dh[i], g @ f[1], rtol=1e-12, atol=1e-15)
            G[i] = g
        np.testing.assert_allclose(dw, G.T @ f[0], rtol=1e-12, atol=1e-15)
        assert math.isclose(loss, float(np.dot(w.astype(np.float64), tl)), rel_tol=1e-12)


def test_fused_gradients_match_finite_differences(oracle):
    """dL/dh_s and dL/dW_s of the fused oracle against central differences of its
    own loss.  Inputs on a grid of 1/32 and steps of 1/256 are exact in bf16."""
    import torch

    rng = np.random.default_rng(15)
    T, d_s, d_t, V = 5, 6, 4, 9
    def q(shape):
        return rng.integers(-16, 17, shape).astype(np.float32) / 32.0
    h_s, W_s, h_t, W_t = q((T, d_s)), q((V, d_s)), q((T, d_t)), q((V, d_t))
    mask = np.array([1, 0, 1, 1, 1], np.uint8)
    w = np.array([0.5, 0.0, 0.25, 1.0, 0.75], np.float32)
    bits = lambda x: W.bf16_bits(torch.from_numpy(x).to(torch.bfloat16))
    def loss(hs, Ws):
        return oracle.fused_lmhead(bits(hs), bits(Ws), bits(h_t), bits(W_t), mask, w)[2]
    dh, _, _, dw = oracle.fused_lmhead(bits(h_s), bits(W_s), bits(h_t), bits(W_t), mask, w, dW=True)
    step = 1.0 / 256
    for (i, c) in [(0, 0), (2, 3), (4, 5), (3, 1)]:
        a, b = h_s.copy(), h_s.copy()
        a[i, c] += step
        b[i, c] -= step
        fd = (loss(a, W_s) - loss(b, W_s)) / (2 * step)
        assert abs(fd - dh[i, c]) <= 1e-4 * max(1.0, np.abs(dh).max()), (i, c, fd, dh[i, c])
    for (v, c) in [(0, 0), (3, 2), (8, 5), (5, 4)]:
        a, b = W_s.copy(), W_s.copy()
        a[v, c] += step
        b[v, c] -= step
        fd = (loss(h_s, a) - loss(h_s, b)) / (2 * step)
        assert abs(fd - dw[v, c]) <= 1e-4 * max(1.0, np.abs(dw).max()), (v, c, fd, dw[v, c])
