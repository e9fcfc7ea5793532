"""GPU parity of the vocabulary-parallel split: shards of one GPU's logits
stand in for ranks (each shard's stats, an ordered merge, each shard's
gradient columns).  The result must match the single-call loss path and the
fp64 oracle at the loss path's bounds; every shard computes bitwise the same
per-token loss."""
import numpy as np
import pytest

import workloads as W
from parity import assert_grad_rows, assert_loss, assert_token_loss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P

    P.load()
    return P


def run_split(P, zs, zt, rot, mask, w, cuts, grad_dtype):
    T = mask.numel()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    parts = torch.empty((len(cuts) - 1, T, 6), dtype=torch.float32, device="cuda")
    ws = torch.empty(max(P.turnopd_loss_workspace_bytes(T), 256), dtype=torch.uint8, device="cuda")
    for r, (a, b) in enumerate(zip(cuts[:-1], cuts[1:])):
        P.turnopd_vocab_shard_stats(zs[:, a:b], zt[:, a:b], rot, mask, parts[r], ws, st)
    merged = torch.empty((T, 6), dtype=torch.float32, device="cuda")
    P.turnopd_vocab_stats_merge(parts, mask, merged)
    grad = torch.full(zs.shape, 7.0, dtype=grad_dtype, device="cuda")
    losses, tls = [], []
    for a, b in zip(cuts[:-1], cuts[1:]):
        tl = torch.empty(T, dtype=torch.float32, device="cuda")
        loss = torch.zeros(1, dtype=torch.float64, device="cuda")
        P.turnopd_vocab_shard_loss_grad(zs[:, a:b], zt[:, a:b], rot, mask, w, merged, grad[:, a:b], 0, tl, loss,
                                        ws, st)
        torch.cuda.synchronize()
        losses.append(loss.item())
        tls.append(tl.cpu().numpy())
    torch.cuda.synchronize()
    assert st.item() == 0
    return grad, tls, losses


@pytest.mark.parametrize("cuts", [[0, 75968, 151936], [0, 50001, 99999, 151936]])
def test_virtual_ranks_match_single_call_and_oracle(P, oracle, cuts):
    b = W.packed(seed=4, num_traj=1, traj_len=1024)
    V = W.V_QWEN
    R = b.num_valid
    zs, zt = W.make_logits(R, V, "agent", torch.bfloat16, seed=40, device="cuda")
    T = b.num_tokens
    rot_np = np.full(T, -1, np.int32)
    rot_np[b.loss_mask == 1] = np.arange(R, dtype=np.int32)
    rot = torch.from_numpy(rot_np).cuda()
    mask = torch.from_numpy(b.loss_mask).cuda()
    w = torch.rand(T, generator=torch.Generator().manual_seed(4)).cuda()
    grad, tls, losses = run_split(P, zs, zt, rot, mask, w, cuts, torch.bfloat16)
    for tl in tls[1:]:
        assert np.array_equal(tl, tls[0])
    assert len(set(losses)) == 1
    # the single-call loss path
    tl1 = torch.empty(T, dtype=torch.float32, device="cuda")
    loss1 = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(P.turnopd_loss_workspace_bytes(T), dtype=torch.uint8, device="cuda")
    P.turnopd_loss_fwd_bwd(zs, zt, V, rot, None, mask, w, 0, None, 0, tl1, loss1, ws, st)
    torch.cuda.synchronize()
    m = b.loss_mask == 1
    assert_token_loss(tls[0][m], tl1.cpu().numpy()[m])
    assert_loss(losses[0], loss1.item())
    # the oracle on a few rows
    toks = np.nonzero(m)[0]
    pick = np.unique(np.concatenate([toks[:2], toks[-2:], np.random.default_rng(0).choice(toks, 3, replace=False)]))
    zsb, ztb = W.bf16_bits(zs), W.bf16_bits(zt)
    g_ref, tl_ref, _ = oracle.loss_fwd_bwd(zsb, ztb, V, b.loss_mask, w.cpu().numpy(), row_of_token=rot_np,
                                           subset=pick)
    assert_token_loss(tls[0][pick], tl_ref[pick])
    rows = rot_np[pick]
    assert_grad_rows(grad.float().cpu().numpy()[rows], g_ref[rows], bf16=True,
                     zs=zs[torch.from_numpy(rows).cuda()], w=w.cpu().numpy()[pick], ell=tl_ref[pick])


def test_fp32_unaligned_split_and_helper(P, oracle):
    """fp32 logits and gradient, a shard boundary that breaks 16-byte alignment,
    and the vocab_parallel_loss helper (a world of one)."""
    from paper_2607_05804_gb300.vocab_parallel import vocab_parallel_loss

    b = W.tiny(seed=2)
    V = 1024
    zs, zt = W.make_logits(b.num_tokens, V, "tiny", torch.float32, seed=41, device="cuda")
    mask = torch.from_numpy(b.loss_mask).cuda()
    w = torch.rand(b.num_tokens, generator=torch.Generator().manual_seed(5)).cuda()
    grad, tls, losses = run_split(P, zs, zt, None, mask, w, [0, 333, 1024], torch.float32)
    g_ref, tl_ref, loss_ref = oracle.loss_fwd_bwd(zs.cpu().numpy(), zt.cpu().numpy(), V, b.loss_mask,
                                                  w.cpu().numpy())
    assert_token_loss(tls[0], tl_ref, b.loss_mask)
    assert_loss(losses[0], loss_ref)
    m = b.loss_mask == 1
    assert_grad_rows(grad.cpu().numpy()[m], g_ref[m], bf16=False)
    tl, loss = vocab_parallel_loss(zs, zt, None, mask, w)
    torch.cuda.synchronize()
    assert_token_loss(tl.cpu().numpy(), tl_ref, b.loss_mask)
    assert_loss(loss.item(), loss_ref)


def test_bad_row_index_sets_status_and_skips_the_token(P, oracle):
    """A supervised token whose row index is out of range: both calls record
    TURNOPD_ERR_TOKEN_RANGE, the token gets loss 0 and no gradient row, and every
    other token matches the oracle with that token masked out."""
    b = W.tiny(seed=3)
    V, T = 1024, b.num_tokens
    zs, zt = W.make_logits(T, V, "tiny", torch.bfloat16, seed=42, device="cuda")
    sup = np.nonzero(b.loss_mask)[0]
    bad = int(sup[len(sup) // 2])
    rot_np = np.arange(T, dtype=np.int32)
    rot_np[bad] = T + 5
    rot = torch.from_numpy(rot_np).cuda()
    mask = torch.from_numpy(b.loss_mask).cuda()
    w = torch.rand(T, generator=torch.Generator().manual_seed(6)).cuda()
    cuts = [0, 512, V]
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(max(P.turnopd_loss_workspace_bytes(T), 256), dtype=torch.uint8, device="cuda")
    parts = torch.empty((2, T, 6), dtype=torch.float32, device="cuda")
    for r, (a, e) in enumerate(zip(cuts[:-1], cuts[1:])):
        P.turnopd_vocab_shard_stats(zs[:, a:e], zt[:, a:e], rot, mask, parts[r], ws, st)
    torch.cuda.synchronize()
    assert st.item() == 5  # TURNOPD_ERR_TOKEN_RANGE
    merged = torch.empty((T, 6), dtype=torch.float32, device="cuda")
    P.turnopd_vocab_stats_merge(parts, mask, merged)
    grad = torch.full(zs.shape, 7.0, dtype=torch.float32, device="cuda")
    tl = torch.full((T,), 3.0, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    for a, e in zip(cuts[:-1], cuts[1:]):
        st.zero_()
        P.turnopd_vocab_shard_loss_grad(zs[:, a:e], zt[:, a:e], rot, mask, w, merged, grad[:, a:e], 0, tl, loss,
                                        ws, st)
        torch.cuda.synchronize()
        assert st.item() == 5
    m2 = b.loss_mask.copy()
    m2[bad] = 0
    g_ref, tl_ref, loss_ref = oracle.loss_fwd_bwd(W.bf16_bits(zs), W.bf16_bits(zt), V, m2, w.cpu().numpy())
    tl_h = tl.cpu().numpy()
    assert tl_h[bad] == 0.0
    assert_token_loss(tl_h, tl_ref, m2)
    assert_loss(loss.item(), loss_ref)
    g = grad.cpu().numpy()
    assert (g[bad] == 7.0).all()  # no token maps to this row
    ok = m2 == 1
    assert_grad_rows(g[ok], g_ref[ok], bf16=False)
