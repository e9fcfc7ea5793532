"""Comparison helpers for GPU-vs-oracle parity tests.

Tolerances (fixed by the target specification of the loss path):
  integer counts, turn ids, offsets      bit-exact
  per-token loss l_i                     |err| <= 1e-4 * max(1, |l_i|)
  total loss                             relative 1e-5
  student-logit gradient, fp32 output    |err| <= 1e-4 * max_v |g_row|
  student-logit gradient, bf16 output    within 2 bf16 ulps of the oracle value, or
                                         within the fp32 bound above (elements far
                                         below the row maximum, where fp32 rounding
                                         of z_s - z_t - c is all that is left)
  sampled-token mode, in addition        g = w l (e_y - p) carries the error of l, which
                                         is bounded absolutely by 1e-4 max(1, |l|) (the
                                         per-token bound): |err_v| may add
                                         w 1e-4 max(1, |l|) |e_y - p_v|
                                         = 1e-4 max(1, |l|) / |l| * |g_v|
  weights (fp32 output of fp64 math)     <= 1 fp32 ulp
  turn-stat sums                         sum of the per-token bounds of the bin
"""
import numpy as np


def assert_weights(w_gpu, w_ref):
    w32 = np.asarray(w_ref, np.float64).astype(np.float32)
    w_gpu = np.asarray(w_gpu, np.float32)
    ulp = np.spacing(np.abs(w32))
    assert (np.abs(w_gpu.astype(np.float64) - w32.astype(np.float64)) <= ulp).all()


def assert_token_loss(tl_gpu, tl_ref, mask=None):
    tl_gpu = np.asarray(tl_gpu, np.float64)
    tl_ref = np.asarray(tl_ref, np.float64)
    err = np.abs(tl_gpu - tl_ref)
    bound = 1e-4 * np.maximum(1.0, np.abs(tl_ref))
    bad = np.nonzero(err > bound)[0]
    assert bad.size == 0, f"{bad.size} tokens off, first {bad[:5]}: {tl_gpu[bad[:5]]} vs {tl_ref[bad[:5]]}"
    if mask is not None:
        assert (tl_gpu[np.asarray(mask) == 0] == 0).all()


def assert_loss(loss_gpu, loss_ref):
    assert abs(loss_gpu - loss_ref) <= 1e-5 * max(abs(loss_ref), 1e-300), (loss_gpu, loss_ref)


def bf16_ulp(x):
    x = np.abs(np.asarray(x, np.float64))
    e = np.floor(np.log2(np.where(x > 0, x, 1.0)))
    return np.where(x > 0, np.exp2(e - 7), 0.0)


def assert_grad_rows(g_gpu, g_ref, bf16: bool, ell=None, w=None):
    """g_gpu, g_ref: [rows, V] float64 arrays of the same rows.  For sampled-token rows
    pass the oracle's per-row loss `ell` and weight `w` (the l-error allowance)."""
    g_gpu = np.asarray(g_gpu, np.float64)
    g_ref = np.asarray(g_ref, np.float64)
    rowmax = np.abs(g_ref).max(axis=1, keepdims=True)
    err = np.abs(g_gpu - g_ref)
    slack = 0.0
    if ell is not None:
        ell = np.asarray(ell, np.float64).reshape(-1, 1)
        w = np.asarray(w, np.float64).reshape(-1, 1)
        lb = 1e-4 * np.maximum(1.0, np.abs(ell))
        slack = np.where(ell != 0, lb / np.where(ell != 0, np.abs(ell), 1.0) * np.abs(g_ref), lb * w)
    err = np.maximum(err - slack, 0.0)
    ok = err <= 1e-4 * rowmax
    if bf16:
        ok |= err <= 2.0 * bf16_ulp(g_ref)
    bad = np.argwhere(~ok)
    assert bad.size == 0, (f"{len(bad)} gradient elements off; first {bad[:3].tolist()}: "
                           f"{g_gpu[tuple(bad[0])]} vs {g_ref[tuple(bad[0])]}")


def assert_stats(st_gpu, st_ref, tl_ref, turn_id, mask, offsets, max_turns):
    B = len(offsets) - 1
    assert np.array_equal(np.asarray(st_gpu["traj_turn_cnt"]).reshape(B, max_turns),
                          st_ref["traj_turn_cnt"])
    assert np.array_equal(np.asarray(st_gpu["turn_cnt"]), st_ref["turn_cnt"])
    assert np.array_equal(np.asarray(st_gpu["turn_surv"]), st_ref["turn_surv"])
    # per-bin bound: sum over its tokens of 1e-4 * max(1, |l_i|)
    bound = np.zeros((B, max_turns))
    tl_ref = np.asarray(tl_ref, np.float64)
    for b in range(B):
        sl = slice(offsets[b], offsets[b + 1])
        m = np.asarray(mask[sl]) == 1
        t = np.asarray(turn_id[sl])[m]
        np.add.at(bound[b], t, 1e-4 * np.maximum(1.0, np.abs(tl_ref[sl][m])))
    tts = np.asarray(st_gpu["traj_turn_sum"]).reshape(B, max_turns)
    assert (np.abs(tts - st_ref["traj_turn_sum"]) <= bound + 1e-12).all()
    assert (np.abs(np.asarray(st_gpu["turn_sum"]) - st_ref["turn_sum"]) <= bound.sum(0) + 1e-12).all()
