"""GPU parity of the fused LM-head path (turnopd_fused_lmhead_fwd_bwd) against
the fp64 oracle.

Tolerances: per-token loss and total loss as for the logit path (the logits are
fp32 tensor-core sums of exact bf16 products instead of fp64 sums: relative
error ~1e-6).  dL/dh_s = G W_s with G rounded to bf16 (2^-9 relative) before
the second product: per element within 1e-2 of its row's maximum |dh|, and a
relative Frobenius error within 4e-3 per row.
"""
import numpy as np
import pytest

import workloads as W
from parity import assert_loss, assert_token_loss

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P

    P.load()
    return P


def assert_dh(dh_gpu, dh_ref):
    dh_gpu = np.asarray(dh_gpu, np.float64)
    dh_ref = np.asarray(dh_ref, np.float64)
    rowmax = np.abs(dh_ref).max(axis=1, keepdims=True)
    err = np.abs(dh_gpu - dh_ref)
    bad = np.argwhere(err > 1e-2 * rowmax + 1e-30)
    assert bad.size == 0, f"{len(bad)} dh elements off, first {bad[:3].tolist()}"
    fro = np.linalg.norm(dh_gpu - dh_ref, axis=1) / np.maximum(np.linalg.norm(dh_ref, axis=1), 1e-30)
    assert (fro <= 4e-3).all(), fro.max()


def run_fused(P, b, d_s, d_t, V, seed, alpha=1.0, grad=True, dw=False):
    from paper_2607_05804_gb300.step import LossStep, to_device

    T = b.num_tokens
    h_s, W_s, h_t, W_t = W.make_fused(T, d_s, d_t, V, seed=seed, device="cuda")
    tid, msk, off, _ = to_device(b, "cuda", compact=False)
    step = LossStep(tid, msk, off, b.max_turns, V, alpha=alpha)
    w = step.weights()
    ws = torch.empty(P.turnopd_fused_workspace_bytes(T, V, d_s, d_t), dtype=torch.uint8, device="cuda")
    dh = torch.full((T, d_s), 3.0, dtype=torch.float32, device="cuda") if grad else None
    dW = torch.full((V, d_s), 5.0, dtype=torch.float32, device="cuda") if dw else None
    tl = torch.full((T,), 7.0, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    P.turnopd_fused_lmhead_fwd_bwd(h_s, W_s, h_t, W_t, msk, w, 0, dh, tl, loss, ws, step.dev_status,
                                   dW_s_out=dW)
    torch.cuda.synchronize()
    assert step.status() == 0
    if dw:
        return (h_s, W_s, h_t, W_t), w.cpu().numpy(), dh, tl.cpu().numpy(), loss.item(), dW
    return (h_s, W_s, h_t, W_t), w.cpu().numpy(), dh, tl.cpu().numpy(), loss.item()


def test_fused_small_all_rows(P, oracle):
    """Ragged vocabulary (1000: last 256-tile partial, padded K 1024) and
    several 128-row tiles with a ragged last tile."""
    b = W.packed(seed=3, num_traj=2, traj_len=160)
    d_s, d_t, V = 256, 192, 1000
    heads, w, dh, tl, loss = run_fused(P, b, d_s, d_t, V, seed=4)
    bits = [W.bf16_bits(x) for x in heads]
    dh_ref, tl_ref, loss_ref = oracle.fused_lmhead(*bits, b.loss_mask, w)
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(loss, loss_ref)
    g = dh.cpu().numpy()
    m = b.loss_mask == 1
    assert (g[~m] == 0).all()
    assert_dh(g[m], dh_ref[m])


def test_fused_forward_only(P, oracle):
    b = W.packed(seed=5, num_traj=1, traj_len=300)
    d_s, d_t, V = 512, 256, 4100
    heads, w, _, tl, loss = run_fused(P, b, d_s, d_t, V, seed=6, grad=False)
    bits = [W.bf16_bits(x) for x in heads]
    _, tl_ref, loss_ref = oracle.fused_lmhead(*bits, b.loss_mask, w)
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(loss, loss_ref)


def test_fused_full_heads_sampled_tokens(P, oracle):
    """Full-size heads (d_s = 4096, d_t = 5120, V = 151,936) on a 600-token batch;
    the oracle recomputes a few supervised tokens, all rows checked by properties."""
    b = W.packed(seed=7, num_traj=1, traj_len=600)
    d_s, d_t, V = 4096, 5120, W.V_QWEN
    heads, w, dh, tl, loss = run_fused(P, b, d_s, d_t, V, seed=8)
    bits = [W.bf16_bits(x) for x in heads]
    valid = np.nonzero(b.loss_mask)[0]
    rng = np.random.default_rng(0)
    pick = np.unique(np.concatenate([valid[:1], valid[-1:], rng.choice(valid, 4, replace=False)]))
    dh_ref, tl_ref, _ = oracle.fused_lmhead(*bits, b.loss_mask, w, subset=pick)
    assert_token_loss(tl[pick], tl_ref[pick])
    g = dh.cpu().numpy()
    assert_dh(g[pick], dh_ref[pick])
    assert (g[b.loss_mask == 0] == 0).all()
    assert (tl[b.loss_mask == 0] == 0).all()
    assert (tl[valid] >= -1e-4).all()
    wl = float(np.dot(w.astype(np.float64), tl.astype(np.float64)))
    assert abs(loss - wl) <= 1e-9 * abs(wl)


def test_fused_all_masked_and_single_row(P, oracle):
    """No supervised row (loss 0, dh zero), then a single supervised row (one
    pair tile holding one valid row)."""
    b = W.packed(seed=11, num_traj=1, traj_len=200)
    b.loss_mask[:] = 0
    heads, w, dh, tl, loss = run_fused(P, b, 256, 64, 700, seed=12)
    assert loss == 0.0
    assert (dh.cpu().numpy() == 0).all() and (tl == 0).all()
    b.loss_mask[57] = 1
    b.turn_id[57] = 0
    heads, w, dh, tl, loss = run_fused(P, b, 256, 64, 700, seed=12)
    bits = [W.bf16_bits(x) for x in heads]
    dh_ref, tl_ref, loss_ref = oracle.fused_lmhead(*bits, b.loss_mask, w)
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(loss, loss_ref)
    g = dh.cpu().numpy()
    assert (np.delete(g, 57, axis=0) == 0).all()
    assert_dh(g[57:58], dh_ref[57:58])


def test_fused_weight_gradient_small(P, oracle):
    """dL/dW_s on a ragged case (V = 1000: partial last vocabulary tile; 305
    supervised rows: partial last token tile) against the oracle, row by row."""
    b = W.packed(seed=3, num_traj=2, traj_len=160)
    d_s, d_t, V = 256, 192, 1000
    heads, w, dh, tl, loss, dW = run_fused(P, b, d_s, d_t, V, seed=4, dw=True)
    bits = [W.bf16_bits(x) for x in heads]
    dh_ref, tl_ref, loss_ref, dw_ref = oracle.fused_lmhead(*bits, b.loss_mask, w, dW=True)
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(loss, loss_ref)
    assert_dh(dh.cpu().numpy()[b.loss_mask == 1], dh_ref[b.loss_mask == 1])
    assert_dh(dW.cpu().numpy(), dw_ref)


def test_fused_weight_gradient_only_and_full_size_identity(P):
    """dW_s without dh_s, then full-size heads: dW_s . W_s and dh_s . h_s both equal
    sum_t,v G[t,v] z_s[t,v] for the same G."""
    b = W.packed(seed=9, num_traj=1, traj_len=600)
    d_s, d_t, V = 4096, 5120, W.V_QWEN
    heads, w, dh, tl, loss, dW = run_fused(P, b, d_s, d_t, V, seed=10, dw=True)
    h_s, W_s = heads[0], heads[1]
    a = float((dW.double() * W_s.double()).sum())
    bsum = float((dh.double() * h_s.double()).sum())
    scale = float((dh.double().abs() * h_s.double().abs()).sum())
    assert abs(a - bsum) <= 2e-3 * scale, (a, bsum, scale)
    heads2, _, dh2, tl2, loss2, dW2 = run_fused(P, b, d_s, d_t, V, seed=10, grad=False, dw=True)
    assert torch.equal(dW2, dW) and loss2 == loss


def test_fused_weight_gradient_all_masked_is_zero(P):
    b = W.packed(seed=11, num_traj=1, traj_len=200)
    b.loss_mask[:] = 0
    heads, w, dh, tl, loss, dW = run_fused(P, b, 256, 64, 700, seed=12, dw=True)
    assert loss == 0.0 and (dW == 0).all()


def test_fused_errors(P):
    T, d_s, d_t, V = 8, 256, 64, 512
    z = lambda *s: torch.zeros(s, dtype=torch.bfloat16, device="cuda")
    msk = torch.ones(T, dtype=torch.uint8, device="cuda")
    w = torch.ones(T, dtype=torch.float32, device="cuda")
    tl = torch.zeros(T, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(P.turnopd_fused_workspace_bytes(T, V, d_s, d_t), dtype=torch.uint8, device="cuda")
    with pytest.raises(P.TurnopdError) as e:  # d_s not a multiple of 256
        P.turnopd_fused_lmhead_fwd_bwd(z(T, 128), z(V, 128), z(T, d_t), z(V, d_t), msk, w, 0, None, tl,
                                       loss, ws, st)
    assert e.value.code == 2
    with pytest.raises(P.TurnopdError) as e:  # sampled mode not offered here
        P.turnopd_fused_lmhead_fwd_bwd(z(T, d_s), z(V, d_s), z(T, d_t), z(V, d_t), msk, w, 1, None, tl,
                                       loss, ws, st)
    assert e.value.code == 6
    with pytest.raises(P.TurnopdError) as e:  # small workspace
        P.turnopd_fused_lmhead_fwd_bwd(z(T, d_s), z(V, d_s), z(T, d_t), z(V, d_t), msk, w, 0, None, tl,
                                       loss, ws[:1024], st)
    assert e.value.code == 10


# Pair tiles are 256 supervised rows; units of the forward and recompute grids are
# enumerated in blocks of at most 16 row tiles; dL/dh_s has (rows/256) x (d_s/256)
# tiles, of which the first floor(tiles/P)*P (P = co-resident pairs, at most 76 on
# 152 SMs) are whole tiles and the rest are split over all pairs.
PAIR_ROWS, UNIT_BLOCK, MAX_PAIRS = 256, 16, 76


def test_fused_mid_size_all_rows_and_weight_gradient(P, oracle):
    """Every supervised row of a 5,255-row batch (21 pair row tiles: the units run
    as two blocks, 11 + 10 row tiles) with d_s = 1024 (84 dh tiles: whole tiles for
    the first 76, split k-ranges and the pair-ordered fixup for the rest), d_t = 256,
    V = 8192 (32 vocabulary tiles: three groups of 10 and a group of 2).  Loss,
    per-token loss, dL/dh_s and dL/dW_s (128 tiles over the pairs, so pairs take two
    tiles through the double accumulator) are compared element by element."""
    b = W.packed(seed=21, num_traj=3, traj_len=2920)
    d_s, d_t, V = 1024, 256, 8192
    m_tiles = -(-b.num_valid // PAIR_ROWS)
    assert m_tiles == 21 and m_tiles > UNIT_BLOCK and m_tiles * (d_s // 256) > MAX_PAIRS
    heads, w, dh, tl, loss, dW = run_fused(P, b, d_s, d_t, V, seed=22, dw=True)
    bits = [W.bf16_bits(x) for x in heads]
    dh_ref, tl_ref, loss_ref, dw_ref = oracle.fused_lmhead(*bits, b.loss_mask, w, dW=True)
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(loss, loss_ref)
    g = dh.cpu().numpy()
    m = b.loss_mask == 1
    assert (g[~m] == 0).all()
    assert_dh(g[m], dh_ref[m])
    assert_dh(dW.cpu().numpy(), dw_ref)


def test_fused_full_size_sampled_rows(P, oracle):
    """The benchmark's fused configuration at full size: 8 x 2048 tokens (9,840
    supervised: 39 pair row tiles, so three unit blocks of 13), d_s = 4096,
    d_t = 5120, V = 151,936, alpha = 1.  The oracle recomputes rows drawn from each
    unit block, from whole dh tiles and from the last row tile, whose 16 dh tiles
    are the split ones; every row is checked by the size-free properties."""
    b = W.fused(0)
    d_s, d_t, V = 4096, 5120, W.V_QWEN
    R = b.num_valid
    m_tiles = -(-R // PAIR_ROWS)
    nb = -(-m_tiles // UNIT_BLOCK)
    mb = -(-m_tiles // nb)
    assert nb == 3 and (m_tiles * (d_s // 256)) % MAX_PAIRS != 0
    heads, w, dh, tl, loss = run_fused(P, b, d_s, d_t, V, seed=30)
    rng = np.random.default_rng(31)
    picks = [0, R - 1]
    for blk in range(nb):                        # rows of every unit block
        lo, hi = blk * mb * PAIR_ROWS, min(R, (blk + 1) * mb * PAIR_ROWS)
        picks += list(rng.integers(lo, hi, 4))
    last = (m_tiles - 1) * PAIR_ROWS            # rows of the split dh tiles
    picks += list(rng.integers(last, R, 4)) + [last]
    rows = np.unique(np.asarray(picks))
    toks = np.nonzero(b.loss_mask)[0][rows]
    bits = [W.bf16_bits(x) for x in heads]
    dh_ref, tl_ref, _ = oracle.fused_lmhead(*bits, b.loss_mask, w, subset=toks)
    assert_token_loss(tl[toks], tl_ref[toks])
    g = dh.cpu().numpy()
    assert_dh(g[toks], dh_ref[toks])
    assert (g[b.loss_mask == 0] == 0).all()
    assert (tl[b.loss_mask == 0] == 0).all()
    assert (tl[b.loss_mask == 1] >= -1e-4).all()
    wl = float(np.dot(w.astype(np.float64), tl.astype(np.float64)))
    assert abs(loss - wl) <= 1e-9 * abs(wl)
