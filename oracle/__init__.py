"""ctypes binding of the fp64 CPU oracle (``turnopd_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test-suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg are the only callers.  The product library never
imports, links or executes anything in this folder, and this folder uses
nothing from the product library.

Arrays are numpy arrays.  bf16 data travels as its raw 16-bit patterns in a
``numpy.uint16`` array (dtype code 1); fp32 data as ``numpy.float32``
(dtype code 0).  Every function returns plain numpy results in float64/int.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import tempfile

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "turnopd_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

F32, BF16 = 0, 1
FULL_VOCAB, SAMPLED_TOKEN = 0, 1
SCOPE_TRAJ, SCOPE_BATCH = 0, 1


class OracleError(RuntimeError):
    def __init__(self, code: int, where: str):
        super().__init__(f"oracle {where} returned status {code}")
        self.code = code


def build(force: bool = False) -> str:
    """Compile liboracle.so beside its source (gcc, -O2, OpenMP, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        fd, tmp = tempfile.mkstemp(suffix=".so", dir=_HERE)
        os.close(fd)
        subprocess.check_call(
            ["gcc", "-O2", "-fopenmp", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


_lib = None


def _L():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
        lib.oracle_turn_counts.argtypes = [P, P, P, i32, i64, i32, P, P]
        lib.oracle_weights.argtypes = [P, P, P, i32, i64, i32, f64, i32, i32, P, P]
        lib.oracle_row.argtypes = [P, P, i32, i64, i32, i32, f64, P, P]
        lib.oracle_loss_fwd_bwd.argtypes = [P, P, i32, i64, i64, P, i64, P, P, P, i64,
                                            i32, P, P, P, P, i64]
        lib.oracle_turn_stats.argtypes = [P, P, P, P, i32, i64, i32, P, P, P, P, P]
        lib.oracle_fused_lmhead.argtypes = [P, P, i64, P, P, i64, i64, P, P, i64, i32,
                                            P, P, P, P, P, P, i64]
        lib.oracle_topk_row.argtypes = [P, P, i32, i64, i32, f64, P, P, P, P]
        lib.oracle_topk_loss.argtypes = [P, P, i32, i64, i64, P, i64, P, P, i64, i32, P, P, P,
                                         P, P, P, i64]
        lib.oracle_alpha_schedule.argtypes = [i64, i64, f64, f64]
        lib.oracle_alpha_schedule.restype = f64
        lib.oracle_num_threads.argtypes = []
        for name in ("oracle_turn_counts", "oracle_weights", "oracle_row",
                     "oracle_loss_fwd_bwd", "oracle_turn_stats", "oracle_fused_lmhead",
                     "oracle_topk_row", "oracle_topk_loss", "oracle_num_threads"):
            getattr(lib, name).restype = ctypes.c_int
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dt):
    return None if a is None else np.ascontiguousarray(a, dtype=dt)


def _check(code, where):
    if code != 0:
        raise OracleError(code, where)


def num_threads() -> int:
    return int(_L().oracle_num_threads())


def _structure(turn_id, loss_mask, traj_offsets):
    return _c(turn_id, np.int32), _c(loss_mask, np.uint8), _c(traj_offsets, np.int64)


def turn_counts(turn_id, loss_mask, traj_offsets, max_turns):
    """-> (n_bt int32[B, max_turns], counts int64[2*max_turns+1] = [S_t, C_t, B'])."""
    tid, msk, off = _structure(turn_id, loss_mask, traj_offsets)
    B, T = off.size - 1, tid.size
    n_bt = np.zeros((max(B, 1), max_turns), np.int32)
    counts = np.zeros(2 * max_turns + 1, np.int64)
    _check(_L().oracle_turn_counts(_p(tid), _p(msk), _p(off), B, T, max_turns,
                                   _p(n_bt), _p(counts)), "turn_counts")
    return n_bt[:B], counts


def weights(turn_id, loss_mask, traj_offsets, max_turns, alpha, scope=SCOPE_TRAJ,
            n_min=0, global_counts=None):
    """Per-token blend weights in float64."""
    tid, msk, off = _structure(turn_id, loss_mask, traj_offsets)
    gc = _c(global_counts, np.int64)
    w = np.zeros(max(tid.size, 1), np.float64)
    _check(_L().oracle_weights(_p(tid), _p(msk), _p(off), off.size - 1, tid.size, max_turns,
                               float(alpha), int(scope), int(n_min), _p(gc), _p(w)), "weights")
    return w[:tid.size]


def _dtype_code(a):
    if a.dtype == np.uint16:
        return BF16
    if a.dtype == np.float32:
        return F32
    raise TypeError("logits must be float32 or uint16 (bf16 bits)")


def row(zs, zt, mode=FULL_VOCAB, y=0, w=1.0, grad=True):
    """One row -> (lse_s, lse_t, l, kl_full, g or None)."""
    zs = np.ascontiguousarray(zs)
    zt = np.ascontiguousarray(zt, dtype=zs.dtype)
    V = zs.size
    out = np.zeros(4, np.float64)
    g = np.zeros(V, np.float64) if grad else None
    _check(_L().oracle_row(_p(zs), _p(zt), _dtype_code(zs), V, int(mode), int(y), float(w),
                           _p(out), _p(g)), "row")
    return out[0], out[1], out[2], out[3], g


def loss_fwd_bwd(zs, zt, vocab, loss_mask, w, mode=FULL_VOCAB, row_of_token=None,
                 sampled_ids=None, grad=True, subset=None):
    """zs, zt: 2-D [R, ld] arrays.  -> (grad [R, V] float64 or None, token_loss, loss)."""
    zs = np.ascontiguousarray(zs)
    zt = np.ascontiguousarray(zt, dtype=zs.dtype)
    R, ld = zs.shape
    msk = _c(loss_mask, np.uint8)
    T = msk.size
    wf = _c(w, np.float32)
    rot = _c(row_of_token, np.int32)
    y = _c(sampled_ids, np.int32)
    sub = _c(subset, np.int64)
    g = np.zeros((R, vocab), np.float64) if grad else None
    tl = np.zeros(max(T, 1), np.float64)
    loss = np.zeros(1, np.float64)
    _check(_L().oracle_loss_fwd_bwd(_p(zs), _p(zt), _dtype_code(zs), ld, vocab, _p(rot), R,
                                    _p(y), _p(msk), _p(wf), T, int(mode), _p(g), _p(tl),
                                    _p(loss), _p(sub), 0 if sub is None else sub.size),
           "loss_fwd_bwd")
    return g, tl[:T], float(loss[0])


def turn_stats(token_loss, turn_id, loss_mask, traj_offsets, max_turns):
    """-> dict of traj_turn_sum [B, Tmax], traj_turn_cnt, turn_sum, turn_cnt, turn_surv."""
    tl = _c(token_loss, np.float64)
    tid, msk, off = _structure(turn_id, loss_mask, traj_offsets)
    B = off.size - 1
    tts = np.zeros((max(B, 1), max_turns), np.float64)
    ttc = np.zeros((max(B, 1), max_turns), np.int32)
    ts = np.zeros(max_turns, np.float64)
    tc = np.zeros(max_turns, np.int64)
    sv = np.zeros(max_turns, np.int32)
    _check(_L().oracle_turn_stats(_p(tl), _p(tid), _p(msk), _p(off), B, tid.size, max_turns,
                                  _p(tts), _p(ttc), _p(ts), _p(tc), _p(sv)), "turn_stats")
    return dict(traj_turn_sum=tts[:B], traj_turn_cnt=ttc[:B], turn_sum=ts, turn_cnt=tc,
                turn_surv=sv)


def fused_lmhead(h_s, W_s, h_t, W_t, loss_mask, w, mode=FULL_VOCAB, sampled_ids=None,
                 subset=None, dW=False):
    """bf16 bit arrays h_s [T, d_s], W_s [V, d_s], h_t [T, d_t], W_t [V, d_t]
    -> (dh_s [T, d_s] float64, token_loss, loss), plus dW_s [V, d_s] float64 last
    when dW is true (over the evaluated tokens)."""
    hs, Ws = _c(h_s, np.uint16), _c(W_s, np.uint16)
    ht, Wt = _c(h_t, np.uint16), _c(W_t, np.uint16)
    T, d_s = hs.shape
    d_t = ht.shape[1]
    V = Ws.shape[0]
    msk = _c(loss_mask, np.uint8)
    wf = _c(w, np.float32)
    y = _c(sampled_ids, np.int32)
    sub = _c(subset, np.int64)
    dh = np.zeros((max(T, 1), d_s), np.float64)
    dw = np.zeros((V, d_s), np.float64) if dW else None
    tl = np.zeros(max(T, 1), np.float64)
    loss = np.zeros(1, np.float64)
    _check(_L().oracle_fused_lmhead(_p(hs), _p(Ws), d_s, _p(ht), _p(Wt), d_t, V, _p(msk),
                                    _p(wf), T, int(mode), _p(y), _p(dh), _p(dw), _p(tl), _p(loss),
                                    _p(sub), 0 if sub is None else sub.size), "fused_lmhead")
    if dW:
        return dh[:T], tl[:T], float(loss[0]), dw
    return dh[:T], tl[:T], float(loss[0])


def topk_row(zs, zt, k_top, w=1.0, grad=True):
    """One row of the teacher top-K reverse KL -> (l, ids [K] int32, g_ids [K] float64,
    dense g [V] float64 or None).  ids are in support order: larger teacher logit first,
    lower id among equal logits."""
    zs = np.ascontiguousarray(zs)
    zt = np.ascontiguousarray(zt, dtype=zs.dtype)
    V = zs.size
    ids = np.zeros(max(int(k_top), 1), np.int32)
    gk = np.zeros(max(int(k_top), 1), np.float64)
    g = np.zeros(V, np.float64) if grad else None
    ell = np.zeros(1, np.float64)
    _check(_L().oracle_topk_row(_p(zs), _p(zt), _dtype_code(zs), V, int(k_top), float(w),
                                _p(ids), _p(gk), _p(g), _p(ell)), "topk_row")
    return float(ell[0]), ids[:k_top], gk[:k_top], g


def topk_loss(zs, zt, vocab, loss_mask, w, k_top, row_of_token=None, grad=False, subset=None):
    """Teacher top-K reverse KL over a batch.  zs, zt: [R, ld].
    -> (topk_ids [T, K] int32, topk_g [T, K] float64, dense grad [R, V] or None,
    token_loss [T], loss); topk rows of unsupervised tokens stay -1 / 0."""
    zs = np.ascontiguousarray(zs)
    zt = np.ascontiguousarray(zt, dtype=zs.dtype)
    R, ld = zs.shape
    msk = _c(loss_mask, np.uint8)
    T = msk.size
    K = int(k_top)
    wf = _c(w, np.float32)
    rot = _c(row_of_token, np.int32)
    sub = _c(subset, np.int64)
    ids = np.full((max(T, 1), max(K, 1)), -1, np.int32)
    gk = np.zeros((max(T, 1), max(K, 1)), np.float64)
    g = np.zeros((R, vocab), np.float64) if grad else None
    tl = np.zeros(max(T, 1), np.float64)
    loss = np.zeros(1, np.float64)
    _check(_L().oracle_topk_loss(_p(zs), _p(zt), _dtype_code(zs), ld, vocab, _p(rot), R,
                                 _p(msk), _p(wf), T, K, _p(ids), _p(gk), _p(g), _p(tl),
                                 _p(loss), _p(sub), 0 if sub is None else sub.size),
           "topk_loss")
    return ids[:T], gk[:T], g, tl[:T], float(loss[0])


def alpha_schedule(k, K, s=0.0, e=1.0) -> float:
    return float(_L().oracle_alpha_schedule(int(k), int(K), float(s), float(e)))
