"""The GPU-vs-oracle comparison helpers (tests/parity.py) on the CPU: a gradient
computed the way an fp32 kernel would (the row's KL off by less than the per-token
bound, then rounded to bf16) passes, and plausible kernel mistakes -- a dropped
KL term, a flipped sign, two swapped columns, an element 3 bf16 ulps off, an
all-zero sampled row whose loss is tiny -- are rejected."""
import numpy as np
import pytest

import oracle
from parity import assert_grad_rows, bf16_ulp

torch = pytest.importorskip("torch")


def _row(seed, V=4096, spike=8.0):
    rng = np.random.default_rng(seed)
    base = rng.normal(0, 3, V)
    zs = base.copy()
    zt = 0.8 * base + 0.6 * rng.normal(0, 3, V)
    ids = rng.choice(V, 5, replace=False)
    zs[ids] += spike
    zt[ids] += spike
    # logits exact in bf16, passed to the oracle as fp32
    zs = torch.tensor(zs).to(torch.bfloat16).float().numpy()
    zt = torch.tensor(zt).to(torch.bfloat16).float().numpy()
    return zs, zt


def _bf16(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16).double().numpy()


def _kernel_like_full(zs, zt, w, dkl):
    """w p (ls - lt - KL') in fp32 with KL' = KL + dkl, rounded to bf16."""
    zs32, zt32 = zs.astype(np.float32), zt.astype(np.float32)
    ls = zs32 - np.float32(np.log(np.exp(zs.astype(np.float64)).sum()))
    lt = zt32 - np.float32(np.log(np.exp(zt.astype(np.float64)).sum()))
    p = np.exp(ls.astype(np.float64)).astype(np.float32)
    kl = np.float32((p.astype(np.float64) * (ls - lt).astype(np.float64)).sum() + dkl)
    return _bf16(np.float32(w) * p * ((ls - lt) - kl)), float(kl)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_full_rows_kernel_like_passes_and_mistakes_fail(seed):
    zs, zt = _row(seed)
    w = 3.0e-4
    _, _, ell, _, g_ref = oracle.row(zs, zt, w=w)
    kw = dict(zs=zs[None, :], w=[w], ell=[ell])
    for dkl in (0.0, 0.5e-4 * max(1.0, abs(ell)), -0.9e-4 * max(1.0, abs(ell))):
        g, _ = _kernel_like_full(zs, zt, w, dkl)
        assert_grad_rows(g[None, :], g_ref[None, :], bf16=True, **kw)
    g, _ = _kernel_like_full(zs, zt, w, 0.0)
    top = int(np.argmax(np.abs(g_ref)))
    mistakes = {
        "dropped KL": _bf16(w * np.exp(zs - np.log(np.exp(zs.astype(np.float64)).sum()))
                            * ((zs - np.log(np.exp(zs.astype(np.float64)).sum()))
                               - (zt - np.log(np.exp(zt.astype(np.float64)).sum())))),
        "sign": np.where(np.arange(g.size) == top, -g, g),
        "swap": g[np.r_[1, 0, 2:g.size]] if g_ref[0] != g_ref[1] else -g,
        "3 ulp": np.where(np.arange(g.size) == top, g + 3 * bf16_ulp(g).numpy(), g),
    }
    for name, bad in mistakes.items():
        with pytest.raises(AssertionError):
            assert_grad_rows(bad[None, :], g_ref[None, :], bf16=True, **kw)


def test_fp32_rows_use_the_row_maximum_bound():
    zs, zt = _row(5)
    _, _, ell, _, g_ref = oracle.row(zs, zt, w=1.0)
    rowmax = np.abs(g_ref).max()
    ok = g_ref + 0.9e-4 * rowmax * np.sign(np.sin(np.arange(g_ref.size)))
    assert_grad_rows(ok[None, :], g_ref[None, :], bf16=False)
    bad = g_ref.copy()
    bad[7] += 1.1e-4 * rowmax
    with pytest.raises(AssertionError):
        assert_grad_rows(bad[None, :], g_ref[None, :], bf16=False)


def test_sampled_rows_follow_the_gpu_loss_even_when_it_is_tiny():
    """g = w l (e_y - p): a tiny l once let any gradient between 0 and 2 g_ref pass."""
    V, y, w = 512, 17, 0.01
    zs, _ = _row(7, V)
    p = np.exp(zs.astype(np.float64) - np.log(np.exp(zs.astype(np.float64)).sum()))
    for ell in (2.5, 3e-6):
        e = np.zeros(V)
        e[y] = 1.0
        g_ref = w * ell * (e - p)
        ell_gpu = ell + 0.5e-4 * max(1.0, ell)
        g_gpu = _bf16(np.float32(w * ell_gpu) * (e - p).astype(np.float32))
        kw = dict(w=[w], ell=[ell], ell_gpu=[ell_gpu], sampled=True)
        info = assert_grad_rows(g_gpu[None, :], g_ref[None, :], bf16=True, **kw)
        assert info["small_ell_rows"] == (1 if ell < 1e-4 else 0)
        with pytest.raises(AssertionError):
            assert_grad_rows(np.zeros((1, V)), g_ref[None, :], bf16=True, **kw)
        with pytest.raises(AssertionError):   # p in place of e_y - p: the sign of every term
            assert_grad_rows(_bf16(np.float32(w * ell_gpu) * p.astype(np.float32))[None, :],
                             g_ref[None, :], bf16=True, **kw)
