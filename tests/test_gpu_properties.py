"""Properties of the CUDA path's outputs that hold by the mathematics of the loss
(Eq. opd-rkl and the turn weights of Sec. 5.2), checked on the GPU results
themselves rather than against the oracle:

  KL(p || p) = 0 and its gradient vanishes;  KL >= 0;
  each gradient row sums to zero (sum_v p_v (ls_v - lt_v - KL) = KL - KL);
  the KL and gradient are invariant to a per-row logit shift and equivariant
  under a permutation of the vocabulary;
  the weights sum to one; at alpha = 1 every non-empty turn of a trajectory
  carries the same mass, at alpha = 0 every trajectory does.

Rows run through the benchmark's launch configuration (V = 151,936 bf16, the
cluster grid beside the helper grid).  Tolerances are those of the parity tests.
"""
import numpy as np
import pytest

import workloads as W
from parity import assert_token_loss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

V = W.V_QWEN


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P

    P.load()
    return P


def run(b, zs, zt, alpha=0.5, grad_dtype=torch.float32):
    from paper_2607_05804_gb300.step import LossStep, to_device

    tid, msk, off, rot = to_device(b, "cuda", True)
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, alpha=alpha)
    grad = torch.full(zs.shape, 7.0, dtype=grad_dtype, device="cuda")
    step.run(zs, zt, grad)
    torch.cuda.synchronize()
    assert step.status() == 0
    T = b.num_tokens
    toks = np.nonzero(b.loss_mask)[0]
    tl = step.token_loss[:T].cpu().numpy()[toks]
    w = step.w[:T].cpu().numpy()[toks]
    return tl, w, grad.double().cpu().numpy()


def dyadic_rows(R, seed):
    """bf16 logits that are multiples of 1/32 in [-3, 3] (the teacher within 1/2 of the
    student), so adding 2 to a row is exact in bf16."""
    g = torch.Generator().manual_seed(seed)
    ks = torch.randint(-96, 97, (R, V), generator=g)
    kt = (ks + torch.randint(-16, 17, (R, V), generator=g)).clamp(-112, 112)
    return (ks.float() / 32).to(torch.bfloat16), (kt.float() / 32).to(torch.bfloat16)


def test_identical_logits_give_zero_kl_and_gradient(P):
    b = W.packed(seed=11, num_traj=1, traj_len=1024)
    zs, _ = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=11, device="cuda")
    tl, w, g = run(b, zs, zs.clone())
    assert np.abs(tl).max() <= 1e-6
    assert np.abs(g).max() <= 1e-6 * w.max()


def test_kl_nonnegative_and_gradient_rows_sum_to_zero(P):
    b = W.packed(seed=12, num_traj=1, traj_len=1024)
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=12, device="cuda")
    tl, w, g = run(b, zs, zt)
    assert (tl >= -1e-6).all()
    assert tl.max() > 0.1  # the teacher differs from the student
    absum = np.abs(g).sum(axis=1)
    assert (np.abs(g.sum(axis=1)) <= 1e-4 * absum).all()


def test_per_row_shift_invariance(P):
    b = W.packed(seed=13, num_traj=1, traj_len=512)
    R = b.num_valid
    zs, zt = dyadic_rows(R, 13)
    zs, zt = zs.cuda(), zt.cuda()
    tl0, _, g0 = run(b, zs, zt)
    shift = torch.zeros((R, 1), dtype=torch.bfloat16, device="cuda")
    shift[::2] = 2.0  # every other row moves by +2 (exact on these values)
    zs1, zt1 = zs + shift, zt + shift
    assert torch.equal((zs1 - shift), zs) and torch.equal((zt1 - shift), zt)
    tl1, _, g1 = run(b, zs1, zt1)
    assert_token_loss(tl1, tl0)
    rowmax = np.abs(g0).max(axis=1, keepdims=True)
    assert (np.abs(g1 - g0) <= 1e-4 * rowmax).all()


def test_vocabulary_permutation(P):
    b = W.packed(seed=14, num_traj=1, traj_len=512)
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=14, device="cuda")
    perm = torch.randperm(V, generator=torch.Generator().manual_seed(14)).cuda()
    tl0, _, g0 = run(b, zs, zt)
    tl1, _, g1 = run(b, zs[:, perm].contiguous(), zt[:, perm].contiguous())
    assert_token_loss(tl1, tl0)
    rowmax = np.abs(g0).max(axis=1, keepdims=True)
    assert (np.abs(g1 - g0[:, perm.cpu().numpy()]) <= 1e-4 * rowmax).all()


@pytest.mark.parametrize("alpha", [0.0, 0.5, 1.0])
def test_weights_sum_to_one_and_balance(P, alpha):
    b = W.household(seed=15)
    from paper_2607_05804_gb300.step import LossStep, to_device

    tid, msk, off, rot = to_device(b, "cuda", True)
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, alpha=alpha)
    step.weights()
    torch.cuda.synchronize()
    assert step.status() == 0
    w = step.w[:b.num_tokens].cpu().numpy().astype(np.float64)
    assert (w[b.loss_mask == 0] == 0).all()
    assert abs(w.sum() - 1.0) <= 1e-5
    offs = b.traj_offsets
    live = [k for k in range(len(offs) - 1) if b.loss_mask[offs[k]:offs[k + 1]].any()]
    for k in live:
        lo, hi = offs[k], offs[k + 1]
        m = b.loss_mask[lo:hi] == 1
        wt, turns = w[lo:hi][m], b.turn_id[lo:hi][m]
        if alpha == 0.0:  # every trajectory the same mass
            assert abs(wt.sum() - 1.0 / len(live)) <= 1e-5 / len(live)
        if alpha == 1.0:  # every non-empty turn of the trajectory the same mass
            ts = np.unique(turns)
            mass = np.array([wt[turns == t].sum() for t in ts])
            target = 1.0 / (len(live) * len(ts))
            assert (np.abs(mass - target) <= 1e-5 * target).all()
