"""Reference (oracle) for the vocabulary-parallel split of the reverse-KL loss
(Eq. opd-rkl): each shard of the vocabulary reduces its columns to per-row
partial statistics, the partials of all shards are merged, and every shard
writes its own columns of the gradient from the merged row constants.

TEST INFRASTRUCTURE ONLY: nothing on the product path imports this module.
float64, plain numpy.  Per row and shard r (columns C_r):
  m_s = max_{C_r} z_s,  S_s = sum_{C_r} e^{z_s - m_s},  A = sum_{C_r} e^{z_s - m_s} (z_s - z_t),
  m_t = max_{C_r} z_t,  S_t = sum_{C_r} e^{z_t - m_t}
merge:  m = max_r m_r,  S = sum_r S_r e^{m_r - m},  A = sum_r A_r e^{m_{s,r} - m_s}
row:    LSE = m + log S,  E_p[z_s - z_t] = A / S_s,  KL = E_p[z_s - z_t] - (LSE_s - LSE_t)
grad:   g_v = w e^{z_s,v - LSE_s} ((z_s - z_t)_v - E_p[z_s - z_t])   for v in C_r
"""
from __future__ import annotations

import numpy as np


def shard_stats(zs, zt):
    """zs, zt: [R, Vr] float64 -> [R, 5] (m_s, S_s, A, m_t, S_t)."""
    zs = np.asarray(zs, np.float64)
    zt = np.asarray(zt, np.float64)
    ms = zs.max(axis=1)
    es = np.exp(zs - ms[:, None])
    mt = zt.max(axis=1)
    et = np.exp(zt - mt[:, None])
    return np.stack([ms, es.sum(axis=1), (es * (zs - zt)).sum(axis=1), mt, et.sum(axis=1)], axis=1)


def merge(parts):
    """parts: [n_shards, R, 5] -> [R, 5], in shard order."""
    parts = np.asarray(parts, np.float64)
    ms = parts[:, :, 0].max(axis=0)
    mt = parts[:, :, 3].max(axis=0)
    fs = np.exp(parts[:, :, 0] - ms)
    ft = np.exp(parts[:, :, 3] - mt)
    return np.stack([ms, (parts[:, :, 1] * fs).sum(axis=0), (parts[:, :, 2] * fs).sum(axis=0), mt,
                     (parts[:, :, 4] * ft).sum(axis=0)], axis=1)


def row_constants(st):
    """merged [R, 5] -> (lse_s, lse_t, e_p, kl)."""
    st = np.asarray(st, np.float64)
    lse_s = st[:, 0] + np.log(st[:, 1])
    lse_t = st[:, 3] + np.log(st[:, 4])
    e_p = st[:, 2] / st[:, 1]
    return lse_s, lse_t, e_p, e_p - (lse_s - lse_t)


def shard_grad(zs, zt, merged, w):
    """Gradient columns of one shard from the merged row statistics."""
    zs = np.asarray(zs, np.float64)
    zt = np.asarray(zt, np.float64)
    lse_s, _, e_p, _ = row_constants(merged)
    p = np.exp(zs - lse_s[:, None])
    return np.asarray(w, np.float64)[:, None] * p * ((zs - zt) - e_p[:, None])
