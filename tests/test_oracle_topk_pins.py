"""Pins of the oracle's teacher top-K reverse KL (the paper's practical loss,
loss_mode topk_reverse_kl, support size K_top; Algorithm 1 "top-K reverse-KL
token losses").  Reading: the support S is the K ids of largest teacher logit,
the lower id first among equal logits, and both distributions are renormalised
over S.  Each pin ties the oracle to something other than itself: the pinned
full-vocabulary KL on a restricted vector, closed forms, invariances, forced
supports, finite differences."""
import math

import numpy as np
import pytest

import oracle


def rng(seed):
    return np.random.default_rng(seed)


def test_k_equals_v_is_the_full_vocabulary_kl():
    r = rng(0)
    V = 257
    zs = r.normal(0, 2, V).astype(np.float32)
    zt = r.normal(0, 2, V).astype(np.float32)
    l, ids, gk, g = oracle.topk_row(zs, zt, V, w=0.7)
    _, _, _, kl, gfull = oracle.row(zs, zt, w=0.7)
    assert abs(l - kl) <= 1e-13 * max(1.0, kl)
    np.testing.assert_allclose(g, gfull, rtol=0, atol=1e-15)
    assert sorted(ids.tolist()) == list(range(V))


def test_uniform_student_spiked_teacher_closed_form_at_k_equals_v():
    V, c = 1000, 6.0
    zs = np.zeros(V, np.float64).astype(np.float32)
    zt = np.zeros(V, np.float32)
    zt[17] = c
    l = oracle.topk_row(zs, zt, V)[0]
    want = -math.log(V) + math.log(math.exp(c) + V - 1) - c / V
    assert abs(l - want) < 1e-12


def test_support_is_renormalised_restriction():
    """zt strictly decreasing in id: S = {0..K-1}; the loss is the full KL of
    the restricted vectors (both renormalised), the gradient is that KL's
    gradient on S and 0 elsewhere."""
    r = rng(1)
    V, K = 300, 50
    zt = (-np.arange(V) * 0.03125).astype(np.float32)
    zs = r.normal(0, 2, V).astype(np.float32)
    l, ids, gk, g = oracle.topk_row(zs, zt, K, w=1.3)
    _, _, _, kl, gsub = oracle.row(zs[:K], zt[:K], w=1.3)
    assert ids.tolist() == list(range(K))
    assert abs(l - kl) <= 1e-13 * max(1.0, kl)
    np.testing.assert_allclose(gk, gsub, rtol=0, atol=1e-15)
    assert (g[K:] == 0).all()
    np.testing.assert_array_equal(g[:K], gk)


def test_support_follows_teacher_not_student():
    V, K = 64, 4
    zs = np.arange(V, dtype=np.float32)          # student prefers high ids
    zt = -np.arange(V, dtype=np.float32)         # teacher prefers low ids
    ids = oracle.topk_row(zs, zt, K)[1]
    assert ids.tolist() == [0, 1, 2, 3]


def test_ties_take_the_lower_id():
    zt = np.array([1, 1, 1, 0, 0, 2, 1], np.float32)
    zs = np.zeros(7, np.float32)
    ids = oracle.topk_row(zs, zt, 3)[1]
    assert ids.tolist() == [5, 0, 1]
    flat = np.zeros(40, np.float32)
    assert oracle.topk_row(flat, flat, 6)[1].tolist() == list(range(6))
    # bf16 input: -0 and +0 are equal logits
    z = np.array([0x8000, 0x0000, 0x8000, 0x3F80], np.uint16)
    assert oracle.topk_row(np.zeros(4, np.uint16), z, 3)[1].tolist() == [3, 0, 1]


@pytest.mark.parametrize("seed", range(6))
def test_selection_equals_a_sort_by_logit_then_id(seed):
    """The support against Python's own sort on (-logit, id), on rows drawn from a
    handful of values (many ties, +0 and -0 among them), for several K."""
    r = rng(100 + seed)
    V = int(r.integers(5, 300))
    levels = np.array([-3.5, -1.0, -0.0, 0.0, 0.25, 2.0, 7.0], np.float32)
    zt = levels[r.integers(0, levels.size, V)]
    zs = r.normal(0, 1, V).astype(np.float32)
    want_all = sorted(range(V), key=lambda v: (-float(zt[v]), v))   # -0.0 == 0.0 as Python floats
    for K in sorted({1, 2, V // 3 + 1, V // 2 + 1, V}):
        ids = oracle.topk_row(zs, zt, K)[1]
        assert ids.tolist() == want_all[:K], (V, K)


def test_off_support_logits_do_not_matter():
    r = rng(2)
    V, K = 500, 20
    zs = r.normal(0, 2, V).astype(np.float32)
    zt = r.normal(0, 2, V).astype(np.float32)
    l, ids, gk, _ = oracle.topk_row(zs, zt, K)
    off = np.setdiff1d(np.arange(V), ids)
    zs2 = zs.copy()
    zs2[off] += r.normal(0, 5, off.size).astype(np.float32)
    zt2 = zt.copy()
    kth = zt[ids[-1]]
    zt2[off] = np.minimum(zt[off] - 1.0, kth - 1.0).astype(np.float32)
    l2, ids2, gk2, _ = oracle.topk_row(zs2, zt2, K)
    assert l2 == l and ids2.tolist() == ids.tolist()
    np.testing.assert_array_equal(gk2, gk)


def test_shift_invariance():
    r = rng(3)
    V, K = 200, 16
    zs = (np.round(r.normal(0, 2, V) * 64) / 64).astype(np.float32)
    zt = (np.round(r.normal(0, 2, V) * 64) / 64).astype(np.float32)
    l, ids, gk, _ = oracle.topk_row(zs, zt, K)
    l2, ids2, gk2, _ = oracle.topk_row(zs + np.float32(3.0), zt - np.float32(5.0), K)
    assert ids2.tolist() == ids.tolist()
    assert abs(l2 - l) <= 1e-13
    np.testing.assert_allclose(gk2, gk, rtol=0, atol=1e-14)


def test_zero_for_identical_models_and_nonnegative():
    r = rng(4)
    V, K = 128, 10
    zt = r.normal(0, 2, V).astype(np.float32)
    l, _, gk, _ = oracle.topk_row(zt, zt, K)
    assert abs(l) < 1e-15 and np.abs(gk).max() < 1e-15
    for s in range(20):
        zs = rng(100 + s).normal(0, 3, V).astype(np.float32)
        assert oracle.topk_row(zs, zt, K)[0] >= -1e-15


def test_two_point_support_bernoulli_closed_form():
    zs = np.array([0.25, -1.5, -9.0, -9.0], np.float32)
    zt = np.array([2.0, 1.0, -3.0, -4.0], np.float32)
    l = oracle.topk_row(zs, zt, 2)[0]
    p = 1.0 / (1.0 + math.exp(-(0.25 - -1.5)))
    q = 1.0 / (1.0 + math.exp(-(2.0 - 1.0)))
    want = p * math.log(p / q) + (1 - p) * math.log((1 - p) / (1 - q))
    assert abs(l - want) < 1e-14


def test_gradient_matches_finite_differences():
    r = rng(5)
    V, K, w = 24, 6, 0.9
    zs = r.normal(0, 1, V)
    zt = r.normal(0, 1, V)
    l, ids, gk, g = oracle.topk_row(zs.astype(np.float32), zt.astype(np.float32), K, w=w)
    # float64 path through float32 inputs: use the exact float32 values
    zs32 = zs.astype(np.float32).astype(np.float64)
    h = 1e-3
    for v in range(V):
        a = zs32.copy(); a[v] += h
        b = zs32.copy(); b[v] -= h
        # dyadic steps keep the float32 inputs exact
        lp = oracle.topk_row(a.astype(np.float32), zt.astype(np.float32), K)[0]
        lm = oracle.topk_row(b.astype(np.float32), zt.astype(np.float32), K)[0]
        ha = (a.astype(np.float32)[v] - b.astype(np.float32)[v]) / 2.0
        fd = w * (lp - lm) / (2.0 * float(ha))
        assert abs(fd - g[v]) <= 2e-5 * max(1.0, abs(g[v])), (v, fd, g[v])


def test_batch_loss_is_weighted_sum_and_masked_rows_untouched():
    r = rng(6)
    T, V, K = 12, 97, 7
    zs = r.normal(0, 2, (T, V)).astype(np.float32)
    zt = r.normal(0, 2, (T, V)).astype(np.float32)
    mask = (r.random(T) < 0.6).astype(np.uint8)
    w = r.random(T).astype(np.float32)
    ids, gk, g, tl, loss = oracle.topk_loss(zs, zt, V, mask, w, K, grad=True)
    assert abs(loss - float(np.dot(w.astype(np.float64), tl))) <= 1e-12
    for i in range(T):
        if mask[i]:
            l1, i1, g1, _ = oracle.topk_row(zs[i], zt[i], K, w=float(w[i]))
            assert tl[i] == l1 and ids[i].tolist() == i1.tolist()
            np.testing.assert_array_equal(gk[i], g1)
            np.testing.assert_array_equal(g[i][i1], g1)
        else:
            assert tl[i] == 0 and (ids[i] == -1).all() and (gk[i] == 0).all() and (g[i] == 0).all()


def test_shape_errors():
    z = np.zeros(8, np.float32)
    with pytest.raises(oracle.OracleError):
        oracle.topk_row(z, z, 9)
    with pytest.raises(oracle.OracleError):
        oracle.topk_row(z, z, 0)
