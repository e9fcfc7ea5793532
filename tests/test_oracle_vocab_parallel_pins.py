"""Pins of the vocabulary-parallel oracle: for any split of the vocabulary,
merging the shards' partial statistics reproduces the full-vocabulary row
oracle (itself pinned by closed forms), and the shard gradients concatenate
to its gradient."""
import numpy as np

import oracle
from oracle import vocab_parallel as VP


def split_points(rng, V, n):
    cuts = np.sort(rng.choice(np.arange(1, V), n - 1, replace=False))
    return [0, *cuts.tolist(), V]


def test_any_split_reproduces_the_full_vocabulary_row():
    rng = np.random.default_rng(0)
    R, V = 6, 301
    zs = rng.normal(0, 2, (R, V)).astype(np.float32)
    zt = rng.normal(0, 2, (R, V)).astype(np.float32)
    w = rng.random(R)
    for n in (1, 2, 3, 7):
        cut = split_points(rng, V, n)
        parts = [VP.shard_stats(zs[:, a:b], zt[:, a:b]) for a, b in zip(cut[:-1], cut[1:])]
        merged = VP.merge(parts)
        lse_s, lse_t, _, kl = VP.row_constants(merged)
        g = np.concatenate([VP.shard_grad(zs[:, a:b], zt[:, a:b], merged, w)
                            for a, b in zip(cut[:-1], cut[1:])], axis=1)
        for r in range(R):
            ls, lt, _, klr, gr = oracle.row(zs[r], zt[r], w=float(w[r]))
            assert abs(lse_s[r] - ls) < 1e-12 and abs(lse_t[r] - lt) < 1e-12
            assert abs(kl[r] - klr) <= 1e-12 * max(1.0, klr)
            np.testing.assert_allclose(g[r], gr, rtol=0, atol=1e-15)


def test_merge_is_order_free_up_to_rounding_and_shift_invariant():
    rng = np.random.default_rng(1)
    zs = rng.normal(0, 3, (4, 100))
    zt = rng.normal(0, 3, (4, 100))
    parts = [VP.shard_stats(zs[:, a:a + 25], zt[:, a:a + 25]) for a in range(0, 100, 25)]
    m1 = VP.merge(parts)
    m2 = VP.merge(parts[::-1])
    np.testing.assert_allclose(VP.row_constants(m1)[3], VP.row_constants(m2)[3], rtol=1e-13)
    shifted = [VP.shard_stats(zs[:, a:a + 25] + 5.0, zt[:, a:a + 25] - 2.0) for a in range(0, 100, 25)]
    np.testing.assert_allclose(VP.row_constants(VP.merge(shifted))[3], VP.row_constants(m1)[3], rtol=1e-12)


def test_one_column_shards_and_peaks_in_different_shards():
    """Every column its own shard, and rows whose student and teacher maxima lie in
    different shards by a wide margin (shards far below the maximum contribute
    e^{m_r - m} ~ 0 and must not disturb the merge)."""
    rng = np.random.default_rng(2)
    R, V = 3, 40
    zs = rng.normal(0, 1, (R, V))
    zt = rng.normal(0, 1, (R, V))
    zs[0, 3] += 80.0          # student peak in column 3
    zt[0, 31] += 60.0         # teacher peak in column 31
    zs[1, :20] -= 700.0       # a whole half far below the other
    zs, zt = zs.astype(np.float32), zt.astype(np.float32)   # the row oracle's input types
    w = np.array([1.0, 0.5, 2.0])
    for cut in ([*range(V + 1)], [0, 4, 30, V], [0, 20, V]):
        parts = [VP.shard_stats(zs[:, a:b], zt[:, a:b]) for a, b in zip(cut[:-1], cut[1:])]
        merged = VP.merge(parts)
        lse_s, lse_t, _, kl = VP.row_constants(merged)
        g = np.concatenate([VP.shard_grad(zs[:, a:b], zt[:, a:b], merged, w)
                            for a, b in zip(cut[:-1], cut[1:])], axis=1)
        assert np.isfinite(kl).all() and np.isfinite(g).all()
        for r in range(R):
            ls, lt, _, klr, gr = oracle.row(zs[r], zt[r], w=float(w[r]))
            assert abs(lse_s[r] - ls) <= 1e-12 * max(1.0, abs(ls))
            assert abs(lse_t[r] - lt) <= 1e-12 * max(1.0, abs(lt))
            assert abs(kl[r] - klr) <= 1e-11 * max(1.0, klr)
            np.testing.assert_allclose(g[r], gr, rtol=0, atol=1e-13 * max(1.0, float(w[r]) * klr))
