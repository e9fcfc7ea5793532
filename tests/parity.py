"""Comparison helpers for GPU-vs-oracle parity tests.

Tolerances (fixed by the target specification of the loss path):
  integer counts, turn ids, offsets      bit-exact
  per-token loss l_i                     |err| <= 1e-4 * max(1, |l_i|)
  total loss                             relative 1e-5
  student-logit gradient, fp32 output    |err| <= 1e-4 * max_v |g_row|
  student-logit gradient, bf16 output    |err| <= 2 bf16 ulps of the oracle value
                                         + w p_v 1e-4 max(1, |l|)   (full vocabulary)
  weights (fp32 output of fp64 math)     <= 1 fp32 ulp
  turn-stat sums                         sum of the per-token bounds of the bin

Why the bf16 bound carries a second term: every element of the full-vocabulary
gradient, g_v = w p_v (ls_v - lt_v - KL), holds the row's KL inside its bracket,
and the per-token bound allows that KL an error of 1e-4 max(1, |KL|); it moves
g_v by w p_v times that much.  Where the bracket nearly cancels (ls_v - lt_v
close to KL) g_v is far smaller than w p_v, and a bound of 2 ulps of g_v alone
would ask the KL to be exact.  Everywhere else the 2-ulp term is the larger
one.  The term is never relative to the row maximum: an element is only
allowed the error that its own probability carries.

Sampled-token rows, g = w l (e_y - p): the loss l carries its own error
(checked by the per-token bound), so the gradient is compared with the
oracle's row rescaled to the GPU's loss, g_ref * l_gpu / l_ref =
w l_gpu (e_y - p), under the plain bound of its dtype.  Rows whose l is
near zero are therefore still held to the shape of e_y - p.

Large arrays are compared with multi-threaded torch CPU float64 operations.
"""
import numpy as np

FLT_MIN = 2.0 ** -126   # below this fp32/bf16 values are subnormal (flushed on the GPU)


def _t(a):
    import torch

    if isinstance(a, torch.Tensor):
        return a.detach().to("cpu", torch.float64)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64))


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
    """Spacing of bf16 numbers at |x| (8 significant bits): 2^(floor(log2|x|) - 7); 0 at 0."""
    import torch

    x = _t(x).abs()
    _, e = torch.frexp(x)                      # x = m 2^e, m in [0.5, 1)
    return torch.exp2((e - 8).to(torch.float64)) * (x > 0)


def probs(zs):
    """Softmax of student logit rows [n, V], in float64 (the scale of the KL allowance)."""
    import torch

    z = _t(zs)
    return torch.exp(z - torch.logsumexp(z, dim=1, keepdim=True))


def assert_grad_rows(g_gpu, g_ref, bf16: bool, *, zs=None, w=None, ell=None, ell_gpu=None,
                     sampled=False):
    """g_gpu, g_ref: [rows, V] arrays of the same rows.

    Full-vocabulary rows in bf16 need the rows' student logits `zs` [rows, V], weights
    `w` and oracle losses `ell` (the KL allowance).  Sampled-token rows need `ell`
    (oracle) and `ell_gpu` (the GPU's token loss), plus `w`.  Returns counts for the
    record: elements compared, bf16 elements beyond 2 ulps (inside the KL allowance),
    and sampled rows with |l| < 1e-4."""
    import torch

    g = _t(g_gpu)
    ref = _t(g_ref)
    n = g.shape[0]
    info = dict(elements=int(g.numel()), beyond_2ulp=0, small_ell_rows=0, max_bracket_err=0.0)
    if sampled:
        ell_r = _t(ell).reshape(n, 1)
        ell_g = _t(ell_gpu).reshape(n, 1)
        ww = _t(w).reshape(n, 1)
        info["small_ell_rows"] = int((ell_r.abs() < 1e-4).sum())
        nz = ell_r != 0
        ref = torch.where(nz, ref * (ell_g / torch.where(nz, ell_r, torch.ones_like(ell_r))), ref)
        # an exactly-zero oracle loss leaves only the magnitude w |l_gpu| |e_y - p| <= w |l_gpu|
        extra = torch.where(nz, torch.zeros_like(ell_r), ww * ell_g.abs())
    else:
        extra = torch.zeros((n, 1), dtype=torch.float64)
    err = (g - ref).abs()
    if not bf16:
        bound = 1e-4 * ref.abs().amax(dim=1, keepdim=True) + extra
    else:
        ulp2 = 2.0 * bf16_ulp(ref)
        bound = ulp2 + extra + FLT_MIN
        if not sampled:
            if zs is None or w is None or ell is None:
                raise ValueError("bf16 full-vocabulary rows need zs, w and ell")
            wp = _t(w).reshape(n, 1) * probs(zs)
            kl_tol = 1e-4 * torch.clamp(_t(ell).reshape(n, 1).abs(), min=1.0)
            bound = bound + wp * kl_tol
            over = err > ulp2 + FLT_MIN
            info["beyond_2ulp"] = int(over.sum())
            if info["beyond_2ulp"]:
                info["max_bracket_err"] = float(((err - ulp2)[over] / wp.expand_as(err)[over]).max())
    bound = bound.expand_as(err)
    ok = err <= bound
    bad = (~ok).nonzero()
    assert bad.shape[0] == 0, (f"{bad.shape[0]} gradient elements off; first {bad[:3].tolist()}: "
                               f"{g[tuple(bad[0])].item()} vs {ref[tuple(bad[0])].item()} "
                               f"(bound {bound[tuple(bad[0])].item()})")
    return info


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
