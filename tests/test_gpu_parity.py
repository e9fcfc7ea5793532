"""GPU parity: libturnopd (through its C ABI) against the fp64 CPU oracle on the
same seeded inputs, element by element, within the tolerances in parity.py.

Sizes: the tiny batch (V = 1024, fp32) exhaustively over alpha x mode x kernel;
packed batches at a reduced vocabulary that spans many tiles and a ragged tail
(every row checked); the three agent-shaped batches at the full V = 151,936 in
bf16 with the benchmark's launch configuration (sampled rows checked against
the oracle, all rows against size-free properties); edge and error cases.
"""
import numpy as np
import pytest

import workloads as W
from parity import (assert_grad_rows, assert_loss, assert_stats, assert_token_loss,
                    assert_weights)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

FORCE_PORTABLE = 0x100
ZERO_MASKED = 0x1


@pytest.fixture(scope="module")
def P():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P

    P.load()
    return P


def make_step(P, b, V, *, compact, mode=0, alpha=0.5, flags=0, y=None, scope=0, n_min=0):
    from paper_2607_05804_gb300.step import LossStep, to_device

    tid, msk, off, rot = to_device(b, "cuda", compact)
    return LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, sampled_ids=y, mode=mode,
                    alpha=alpha, scope=scope, n_min=n_min, flags=flags)


def per_token_ids(b, y_rows, compact):
    """Sampled ids are per token; for compact rows, row k belongs to the k-th supervised token."""
    if not compact:
        return y_rows
    y = torch.zeros(b.num_tokens, dtype=torch.int32, device=y_rows.device)
    idx = torch.from_numpy(np.nonzero(b.loss_mask)[0]).to(y_rows.device)
    y[idx] = y_rows
    return y


def bits_or_f32(z):
    return W.bf16_bits(z) if z.dtype == torch.bfloat16 else z.detach().cpu().numpy()


def run_chain(P, oracle, b, V, zs, zt, *, mode, alpha, flags=0, grad_dtype=None, compact=False,
              scope=0, n_min=0, seed_y=1, y_rel=None):
    """GPU chain vs oracle chain on every row of the batch.  y_rel (sampled mode): also
    hold each row's g_y = w l (1 - p_y) to y_rel of the oracle's (after the l rescaling);
    returns the oracle's 1 - p_y of the rows as a third value then."""
    y = per_token_ids(b, W.sample_ids(zs, seed_y, V), compact) if mode == 1 else None
    step = make_step(P, b, V, compact=compact, mode=mode, alpha=alpha, flags=flags, y=y,
                     scope=scope, n_min=n_min)
    gdt = zs.dtype if grad_dtype is None else grad_dtype
    grad = torch.full(zs.shape, 7.0, dtype=gdt, device="cuda")
    step.run(zs, zt, grad)
    torch.cuda.synchronize()
    assert step.status() == 0
    T = b.num_tokens
    w_ref = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, alpha, scope, n_min)
    w_gpu = step.w[:T].cpu().numpy()
    assert_weights(w_gpu, w_ref)
    rot = b.compact_rows() if compact else None
    ynp = y.cpu().numpy() if y is not None else None
    g_ref, tl_ref, loss_ref = oracle.loss_fwd_bwd(
        bits_or_f32(zs), bits_or_f32(zt), V, b.loss_mask, w_ref.astype(np.float32), mode=mode,
        row_of_token=rot, sampled_ids=ynp)
    tl = step.token_loss[:T].cpu().numpy()
    assert_token_loss(tl, tl_ref, b.loss_mask)
    assert_loss(step.loss.item(), loss_ref)
    rows = np.nonzero(b.loss_mask)[0] if not compact else np.arange(b.num_valid)
    toks = np.nonzero(b.loss_mask)[0]
    g = grad.float().cpu().numpy().astype(np.float64)
    rsel = torch.from_numpy(rows).to(zs.device)
    assert_grad_rows(g[rows][:, :V], g_ref[rows], bf16=(gdt == torch.bfloat16),
                     zs=zs[rsel, :V], w=w_ref.astype(np.float32)[toks], ell=tl_ref[toks],
                     ell_gpu=tl[toks], sampled=(mode == 1))
    omp = None
    if y_rel is not None:
        assert mode == 1
        yk = ynp[toks].astype(np.int64)
        gy, gy_ref = g[rows, yk], g_ref[rows, yk]
        wl_ref = w_ref.astype(np.float32)[toks].astype(np.float64) * tl_ref[toks]
        nz = wl_ref != 0
        omp = gy_ref[nz] / wl_ref[nz]
        ref = gy_ref[nz] * (tl[toks][nz] / tl_ref[toks][nz])
        err = np.abs(gy[nz] - ref)
        assert (err <= y_rel * np.abs(ref)).all(), (
            f"g_y off: worst relative {float((err / np.abs(ref)).max()):.3g} at 1 - p_y = "
            f"{float(omp[np.argmax(err / np.abs(ref))]):.3g}")
    st_ref = oracle.turn_stats(tl_ref, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    st = {k: v.cpu().numpy() for k, v in step.stats().items()}
    assert_stats(st, st_ref, tl_ref, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    if y_rel is not None:
        return step, grad, omp
    return step, grad


# ---------------------------------------------------------------- tiny batch, exhaustive

@pytest.mark.parametrize("flags", [0, FORCE_PORTABLE], ids=["default", "portable"])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
@pytest.mark.parametrize("alpha", [0.0, 0.5, 1.0])
def test_tiny_exhaustive(P, oracle, alpha, mode, flags):
    b = W.tiny()
    zs, zt = W.make_logits(b.num_tokens, 1024, "tiny", torch.float32, seed=0, device="cuda")
    run_chain(P, oracle, b, 1024, zs, zt, mode=mode, alpha=alpha, flags=flags)


# ---------------------------------------------------------------- reduced vocabulary, all rows

@pytest.mark.parametrize("V,ld", [(4099, 4104), (4099, 4099), (16384, 16384)])
@pytest.mark.parametrize("gdt", ["bf16", "f32"])
@pytest.mark.parametrize("flags", [0, FORCE_PORTABLE], ids=["default", "portable"])
@pytest.mark.parametrize("idt", ["bf16", "f32"])
def test_packed_reduced_vocab(P, oracle, V, ld, gdt, flags, idt):
    b = W.packed(seed=2, num_traj=4, traj_len=1024)
    zs, zt = W.make_logits(b.num_tokens, V, "agent", torch.bfloat16 if idt == "bf16" else torch.float32,
                           seed=3, device="cuda", ld=ld)
    run_chain(P, oracle, b, V, zs, zt, mode=0, alpha=0.5, flags=flags,
              grad_dtype=torch.bfloat16 if gdt == "bf16" else torch.float32)


@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
def test_household_compact_reduced_vocab(P, oracle, mode):
    b = W.household(seed=5, num_traj=4, traj_len=4096)
    V = 8192
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=6, device="cuda")
    run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.25, compact=True)


@pytest.mark.parametrize("scope,n_min", [(0, 2), (1, 0), (1, 3)])
def test_scopes_and_floor(P, oracle, scope, n_min):
    b = W.multihop(seed=7, num_traj=6, min_len=256, max_len=2048)
    V = 2048
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=8, device="cuda")
    run_chain(P, oracle, b, V, zs, zt, mode=0, alpha=0.7, compact=True, scope=scope, n_min=n_min)


def test_paper_turn_floor_on_household(P, oracle):
    """The paper's internal-blend floor, n_min = max(8, ceil(0.15 n_traj)) = 8 for the
    16 household trajectories, whose deep turn indices have 7 survivors or fewer:
    the weights of the whole batch for alpha in {0.5, 1}, then the chain on every
    row of a shorter household batch (turns 9 and 10 below the floor)."""
    b = W.household(0)
    n_min = P.turnopd_turn_floor(b.num_traj)
    assert n_min == 8
    _, counts = oracle.turn_counts(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    surv = counts[:b.max_turns]
    assert ((surv > 0) & (surv < n_min)).any() and (surv >= n_min).any()
    for alpha in (0.5, 1.0):
        step = make_step(P, b, 8, compact=True, alpha=alpha, n_min=n_min)
        step.weights()
        torch.cuda.synchronize()
        assert step.status() == 0
        assert_weights(step.w[:b.num_tokens].cpu().numpy(),
                       oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, alpha,
                                      n_min=n_min))
    b = W.household(seed=5, num_traj=16, traj_len=2048)
    V = 4096
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=9, device="cuda")
    run_chain(P, oracle, b, V, zs, zt, mode=0, alpha=1.0, compact=True,
              n_min=P.turnopd_turn_floor(b.num_traj))


# ---------------------------------------------------------------- cluster kernel, all rows

@pytest.mark.parametrize("V", [8192, 32000, 50000, W.V_QWEN, 200000, 262144])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
@pytest.mark.parametrize("gdt", ["bf16", "f32"])
def test_cluster_kernel_all_rows(P, oracle, V, mode, gdt):
    """The bf16 row path on every row (vocabulary a multiple of 8): V = 8,192 takes the
    helper kernel alone, V = 32,000 clusters of 2 on every SM, V = 50,000 clusters of 3
    beside the helper (ragged last slice), V = 151,936 clusters of 8 beside it, and
    V = 200,000 and 262,144 clusters of 16 beside it (200,000: slices of 1,563 vectors,
    the shortest the clusters of 16 take)."""
    b = W.packed(seed=11, num_traj=2, traj_len=256)
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=12, device="cuda")
    run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.5, compact=True,
              grad_dtype=torch.bfloat16 if gdt == "bf16" else torch.float32)


@pytest.mark.parametrize("kernel,V,idt,flags", [
    ("helper alone", 8192, "bf16", 0), ("clusters of 2", 32000, "bf16", 0),
    ("clusters of 8 + helper", W.V_QWEN, "bf16", 0), ("split rows", 4100, "f32", 0),
    ("split rows", W.V_QWEN, "f32", 0), ("portable", 4099, "bf16", FORCE_PORTABLE),
    ("portable", 4100, "f32", FORCE_PORTABLE)])
@pytest.mark.parametrize("gdt", ["bf16", "f32"])
def test_sampled_peaked_rows(P, oracle, kernel, V, idt, flags, gdt):
    """Sampled-token rows whose student logit at y stands delta = 0 ... 30 above the rest
    of the row, so that p_y runs from ordinary values to within ~1e-9 of 1: every row
    path keeps g_y = w l (1 - p_y) to fp32 relative precision (a gradient formed as
    w l - w l p_y keeps no digit of it there).  Raising z_s at the Gumbel-max sample
    keeps it the sample, so run_chain draws the same y."""
    b = W.packed(seed=41, num_traj=2, traj_len=256)
    dt = torch.bfloat16 if idt == "bf16" else torch.float32
    zs, zt = W.make_logits(b.num_valid, V, "agent", dt, seed=42, device="cuda")
    y = W.sample_ids(zs, 43, V).long()
    r = torch.arange(b.num_valid, device="cuda")
    delta = torch.tensor([0.0, 3.0, 6.0, 10.0, 15.0, 20.0, 25.0, 30.0], device="cuda")[r % 8]
    zs[r, y] = (zs[:, :V].float().amax(dim=1) + delta).to(dt)
    assert torch.equal(W.sample_ids(zs, 43, V).long(), y)
    gd = torch.bfloat16 if gdt == "bf16" else torch.float32
    out = run_chain(P, oracle, b, V, zs, zt, mode=1, alpha=0.5, flags=flags, compact=True,
                    grad_dtype=gd, seed_y=43, y_rel=(1e-4 if gdt == "f32" else 2.0 ** -7))
    assert out[2].min() < 1e-8  # the test reaches p_y within 1e-8 of 1


@pytest.mark.parametrize("V,ld", [(4100, 4100), (4100, 4104), (W.V_QWEN, W.V_QWEN), (262144, 262144)])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
@pytest.mark.parametrize("gdt", ["bf16", "f32"])
def test_split_kernel_fp32_all_rows(P, oracle, V, ld, mode, gdt):
    """fp32 logits through the split-row kernel on every row: clusters of 4 CTAs
    share each row (ragged last slice at V = 4100, a ragged last chunk at
    V = 151,936, whole chunks at 262,144), about 8 rows per cluster so the chunk
    ring wraps across rows, and padding columns beyond V never read."""
    b = W.packed(seed=11, num_traj=2, traj_len=256)
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.float32, seed=12, device="cuda", ld=ld)
    _, grad = run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.5, compact=True,
                        grad_dtype=torch.bfloat16 if gdt == "bf16" else torch.float32)
    if ld > V:
        assert (grad[:, V:].float() == 7.0).all()


@pytest.mark.parametrize("ld", [151937, 151944])
@pytest.mark.parametrize("idt", ["bf16", "f32"])
def test_odd_vocabulary_full_size(P, oracle, ld, idt):
    """V = 151,937 (not a multiple of 8 or 4) at the full size, with a row stride that
    breaks 16-byte alignment and one padded to a multiple of 8: every row through the
    kernel these shapes take, the padding columns of the gradient never written."""
    b = W.packed(seed=31, num_traj=1, traj_len=256)
    V = 151937
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16 if idt == "bf16" else torch.float32,
                           seed=32, device="cuda", ld=ld)
    for mode in (0, 1):
        _, grad = run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.5, compact=True)
        if ld > V:
            assert (grad[:, V:].float() == 7.0).all()


@pytest.mark.parametrize("V", [8193, 32007, 50005, W.V_QWEN + 1, W.V_QWEN + 7])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
@pytest.mark.parametrize("gdt", ["bf16", "f32"])
def test_masked_tail_vocab(P, oracle, V, mode, gdt):
    """bf16 rows with V % 8 != 0 and the stride padded to a multiple of 8 take the row
    grids with a masked last vector: V = 8,193 the helper alone, 32,007 clusters of 2,
    50,005 clusters of 3 beside the helper, 151,937 and 151,943 clusters of 8 beside it.
    NaN and inf fill the padding; its gradient columns stay untouched.  In sampled mode
    every third row's y is pushed into the masked vector (its student logit 30 above the
    row, so the Gumbel-max draw picks it)."""
    b = W.packed(seed=51, num_traj=2, traj_len=256)
    ld = (V + 7) // 8 * 8
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=52, device="cuda", ld=ld)
    if mode == 1:
        r = torch.arange(0, b.num_valid, 3, device="cuda")
        zs[r, V - 1] = (zs[r, :V].float().amax(dim=1) + 30.0).to(torch.bfloat16)
    zs[:, V:] = float("nan")
    zt[:, V:] = float("inf")
    _, grad = run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.5, compact=True, seed_y=53,
                        grad_dtype=torch.bfloat16 if gdt == "bf16" else torch.float32)
    assert (grad[:, V:].float() == 7.0).all()
    if mode == 1:
        y = W.sample_ids(zs, 53, V)
        assert (y[r] == V - 1).all()


@pytest.mark.parametrize("n_sup", [1, 5])
def test_split_kernel_fewer_rows_than_clusters(P, oracle, n_sup):
    """fp32 rows at the full vocabulary with fewer rows than clusters: most clusters
    have no row and leave at once."""
    T = 40
    turn_id = np.full(T, -1, np.int32)
    mask = np.zeros(T, np.uint8)
    idx = np.linspace(3, T - 2, n_sup).astype(int)
    mask[idx] = 1
    turn_id[idx] = np.arange(n_sup) % 3
    b = W.Batch("few", turn_id, mask, np.array([0, T], np.int64), 3)
    zs, zt = W.make_logits(b.num_valid, FULL_V, "agent", torch.float32, seed=60 + n_sup, device="cuda")
    for mode in (0, 1):
        run_chain(P, oracle, b, FULL_V, zs, zt, mode=mode, alpha=0.5, compact=True,
                  grad_dtype=torch.float32)


@pytest.mark.parametrize("V", [50000, W.V_QWEN])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
def test_forward_only_all_rows(P, oracle, V, mode):
    """No gradient buffer: the loss and every token's l through both row grids (the
    clusters' share of the rows and the helper grid's)."""
    b = W.packed(seed=17, num_traj=2, traj_len=512)
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=17, device="cuda")
    y = per_token_ids(b, W.sample_ids(zs, 3, V), True) if mode == 1 else None
    step = make_step(P, b, V, compact=True, mode=mode, alpha=0.5, y=y)
    step.run(zs, zt, None)
    torch.cuda.synchronize()
    assert step.status() == 0
    T = b.num_tokens
    w_ref = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, 0.5)
    _, tl_ref, loss_ref = oracle.loss_fwd_bwd(
        bits_or_f32(zs), bits_or_f32(zt), V, b.loss_mask, w_ref.astype(np.float32), mode=mode,
        row_of_token=b.compact_rows(), sampled_ids=y.cpu().numpy() if y is not None else None, grad=False)
    assert_token_loss(step.token_loss[:T].cpu().numpy(), tl_ref, b.loss_mask)
    assert_loss(step.loss.item(), loss_ref)


@pytest.mark.parametrize("n_sup", [1, 2, 3, 7])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
def test_few_rows_split_between_grids(P, oracle, n_sup, mode):
    """A handful of supervised rows at the full vocabulary: the row list's cut leaves
    the cluster grid none or a few of them and the helper grid the rest."""
    T = 40
    turn_id = np.full(T, -1, np.int32)
    mask = np.zeros(T, np.uint8)
    idx = np.linspace(3, T - 2, n_sup).astype(int)
    mask[idx] = 1
    turn_id[idx] = np.arange(n_sup) % 3
    b = W.Batch("few", turn_id, mask, np.array([0, T], np.int64), 3)
    V = FULL_V
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=40 + n_sup, device="cuda")
    run_chain(P, oracle, b, V, zs, zt, mode=mode, alpha=0.5, compact=True)


def test_cluster_matches_portable(P, oracle):
    """Both kernels agree with each other to within the oracle tolerances."""
    b = W.packed(seed=13, num_traj=2, traj_len=512)
    V = W.V_QWEN
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=13, device="cuda")
    out = []
    for flags in (0, FORCE_PORTABLE):
        step = make_step(P, b, V, compact=True, flags=flags)
        g = torch.empty(zs.shape, dtype=torch.float32, device="cuda")
        step.run(zs, zt, g)
        torch.cuda.synchronize()
        assert step.status() == 0
        out.append((g, step.token_loss[:b.num_tokens].clone(), step.loss.item()))
    (g0, t0, l0), (g1, t1, l1) = out
    assert abs(l0 - l1) <= 2e-5 * abs(l0)
    assert ((t0 - t1).abs() <= 2e-4 * t0.abs().clamp(min=1)).all()
    rowmax = g0.abs().amax(dim=1, keepdim=True)
    assert ((g0 - g1).abs() <= 2e-4 * rowmax).all()


# ---------------------------------------------------------------- full vocabulary, sampled rows

FULL_V = W.V_QWEN


def full_size_check(P, oracle, b, mode, alpha, seed=0, chunk=256):
    """The batch at V = 151,936 bf16 through the benchmark's launch configuration,
    every supervised row against the oracle: per-token loss, the gradient row, the
    total loss and the turn statistics.  Returns the comparison counts."""
    V = FULL_V
    R = b.num_valid
    zs, zt = W.make_logits(R, V, "agent", torch.bfloat16, seed=seed, device="cuda")
    y_rows = W.sample_ids(zs, seed + 1) if mode == 1 else None
    y = per_token_ids(b, y_rows, True) if mode == 1 else None
    step = make_step(P, b, V, compact=True, mode=mode, alpha=alpha, y=y)
    grad = torch.empty_like(zs)
    step.run(zs, zt, grad)
    torch.cuda.synchronize()
    assert step.status() == 0
    T = b.num_tokens
    w_ref = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, alpha)
    assert_weights(step.w[:T].cpu().numpy(), w_ref)
    w32 = w_ref.astype(np.float32)
    tl = step.token_loss[:T].cpu().numpy()
    toks_all = np.nonzero(b.loss_mask)[0]
    y_np = y_rows.cpu().numpy() if y_rows is not None else None
    tl_ref = np.zeros(T, np.float64)
    totals = dict(elements=0, beyond_2ulp=0, small_ell_rows=0, max_bracket_err=0.0)
    for r0 in range(0, R, chunk):
        r1 = min(R, r0 + chunk)
        n = r1 - r0
        toks = toks_all[r0:r1]
        g_ref, t_ref, _ = oracle.loss_fwd_bwd(
            W.bf16_bits(zs[r0:r1]), W.bf16_bits(zt[r0:r1]), V, np.ones(n, np.uint8), w32[toks],
            mode=mode, row_of_token=np.arange(n, dtype=np.int32),
            sampled_ids=y_np[r0:r1] if y_np is not None else None)
        tl_ref[toks] = t_ref
        assert_token_loss(tl[toks], t_ref)
        info = assert_grad_rows(grad[r0:r1], g_ref, bf16=True, zs=zs[r0:r1], w=w32[toks], ell=t_ref,
                                ell_gpu=tl[toks], sampled=(mode == 1))
        for k in ("elements", "beyond_2ulp", "small_ell_rows"):
            totals[k] += info[k]
        totals["max_bracket_err"] = max(totals["max_bracket_err"], info["max_bracket_err"])
    assert (tl[b.loss_mask == 0] == 0).all()
    # L = sum_i w_i l_i over the oracle's l (Eq. opd-rkl with the blend weights)
    assert_loss(step.loss.item(), float(np.dot(w32.astype(np.float64), tl_ref)))
    st_ref = oracle.turn_stats(tl_ref, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    st = {k: v.cpu().numpy() for k, v in step.stats().items()}
    assert_stats(st, st_ref, tl_ref, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
    print(f"\nfull-size parity {b.name} mode={mode}: rows={R} elements={totals['elements']} "
          f"bf16 beyond 2 ulp={totals['beyond_2ulp']} "
          f"(max bracket error {totals['max_bracket_err']:.3g}) "
          f"sampled rows |l|<1e-4={totals['small_ell_rows']}")
    return totals


def test_full_packed(P, oracle):
    full_size_check(P, oracle, W.packed(0), mode=0, alpha=0.5)


def test_full_household(P, oracle):
    for alpha in (0.0, 0.25, 0.5, 0.75, 1.0):
        b = W.household(0)
        V = FULL_V
        # weights over the full batch for every alpha of the sweep
        step = make_step(P, b, V, compact=True, alpha=alpha)
        step.weights()
        torch.cuda.synchronize()
        assert step.status() == 0
        assert_weights(step.w[:b.num_tokens].cpu().numpy(),
                       oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, alpha))
    full_size_check(P, oracle, W.household(0), mode=0, alpha=0.5, seed=3)


@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
def test_full_multihop(P, oracle, mode):
    full_size_check(P, oracle, W.multihop(0), mode=mode, alpha=0.5, seed=5)


# ---------------------------------------------------------------- turn stats in isolation

def test_turn_stats_full_size(P, oracle):
    from paper_2607_05804_gb300.step import to_device

    for b in (W.household(0), W.multihop(0)):
        rng = np.random.default_rng(3)
        tl = (rng.gamma(2.0, 1.0, b.num_tokens) * b.loss_mask).astype(np.float32)
        step = make_step(P, b, 8, compact=True)
        step.token_loss[:b.num_tokens] = torch.from_numpy(tl).cuda()
        step.turn_stats()
        torch.cuda.synchronize()
        assert step.status() == 0
        st_ref = oracle.turn_stats(tl.astype(np.float64), b.turn_id, b.loss_mask, b.traj_offsets,
                                   b.max_turns)
        st = {k: v.cpu().numpy() for k, v in step.stats().items()}
        assert np.array_equal(st["traj_turn_cnt"], st_ref["traj_turn_cnt"])
        assert np.array_equal(st["turn_cnt"], st_ref["turn_cnt"])
        assert np.array_equal(st["turn_surv"], st_ref["turn_surv"])
        np.testing.assert_allclose(st["traj_turn_sum"], st_ref["traj_turn_sum"], rtol=1e-12, atol=1e-9)
        np.testing.assert_allclose(st["turn_sum"], st_ref["turn_sum"], rtol=1e-12, atol=1e-9)


# ---------------------------------------------------------------- edge and error cases

def test_empty_and_all_masked(P, oracle):
    from paper_2607_05804_gb300.step import LossStep

    # empty batch
    e = lambda dt: torch.zeros(0, dtype=dt, device="cuda")
    off = torch.zeros(2, dtype=torch.int64, device="cuda")
    step = LossStep(e(torch.int32), e(torch.uint8), off, 3, 16)
    z = torch.zeros((0, 16), dtype=torch.bfloat16, device="cuda")
    step.loss.fill_(5.0)
    step.run(z, z, torch.zeros_like(z))
    torch.cuda.synchronize()
    assert step.status() == 0 and step.loss.item() == 0.0
    # all-masked batch with empty trajectories
    b = W._from_spans("masked", [[("o", 40)], [], [("o", 7), ("p", 3)]], max_turns=2)
    zs, zt = W.make_logits(b.num_tokens, 64, "tiny", torch.float32, seed=0, device="cuda")
    step = make_step(P, b, 64, compact=False)
    step.token_loss.fill_(3.0)
    step.run(zs, zt, torch.zeros_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 0
    assert step.loss.item() == 0.0
    assert not step.w.any() and not step.token_loss.any()
    assert not step.turn_cnt.any()


def test_random_structures_with_empty_trajectories(P, oracle):
    rng = np.random.default_rng(42)
    for k in range(6):
        b = W.random_structure(rng, num_traj=int(rng.integers(1, 9)), max_len=80,
                               max_turns=int(rng.integers(1, 7)))
        zs, zt = W.make_logits(b.num_tokens, 40, "agent", torch.bfloat16, seed=k, device="cuda",
                               ld=48)
        if b.num_tokens == 0:
            continue
        run_chain(P, oracle, b, 40, zs, zt, mode=k % 2, alpha=0.3 * (k % 4))


@pytest.mark.parametrize("ld,gdt", [(1024, torch.bfloat16), (1003, torch.bfloat16), (1001, torch.float32)])
def test_zero_masked_grad_and_untouched_rows(P, oracle, ld, gdt):
    """Masked rows are zeroed only with the flag; odd row strides put the row starts off
    16-byte boundaries (the zero fill's element-wise head and tail)."""
    b = W.packed(seed=4, num_traj=2, traj_len=512)
    V = 1000
    zs, zt = W.make_logits(b.num_tokens, V, "agent", torch.bfloat16, seed=4, device="cuda", ld=ld)
    for flags in (0, ZERO_MASKED):
        step = make_step(P, b, V, compact=False, flags=flags)
        grad = torch.full(zs.shape, 3.0, dtype=gdt, device="cuda")
        step.run(zs, zt, grad)
        torch.cuda.synchronize()
        masked = torch.from_numpy(b.loss_mask == 0).cuda()
        g = grad[masked]
        if flags:
            assert not g[:, :V].any()
        else:
            assert (g[:, :V] == 3.0).all()
        assert (grad[:, V:] == 3.0).all()  # padding columns never written


def test_padding_never_read(P, oracle):
    """NaN and inf in the padding columns change no bit of any result (V = 500: the bf16
    row path reads the last vector's padding up to column 504 and masks it)."""
    b = W.packed(seed=6, num_traj=2, traj_len=256)
    V = 500
    zs, zt = W.make_logits(b.num_tokens, V, "agent", torch.bfloat16, seed=6, device="cuda", ld=512)
    ref_step, ref_grad = run_chain(P, oracle, b, V, zs, zt, mode=0, alpha=0.5)
    zs[:, V:] = float("nan")
    zt[:, V:] = float("inf")
    step = make_step(P, b, V, compact=False)
    grad = torch.full(zs.shape, 7.0, dtype=torch.bfloat16, device="cuda")
    step.run(zs, zt, grad)
    torch.cuda.synchronize()
    assert step.status() == 0
    assert torch.equal(grad, ref_grad) and step.loss.item() == ref_step.loss.item()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_deterministic(P, oracle, dtype):
    """Two calls on the same inputs give the same bits (fixed merge orders in the
    cluster kernel and helper grid for bf16, in the split-row clusters for fp32)."""
    b = W.packed(seed=1, num_traj=4, traj_len=2048)
    V = FULL_V
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16 if dtype == "bf16" else torch.float32,
                           seed=1, device="cuda")
    outs = []
    for _ in range(2):
        step = make_step(P, b, V, compact=True)
        grad = torch.empty_like(zs)
        step.run(zs, zt, grad)
        torch.cuda.synchronize()
        outs.append((grad.clone(), step.token_loss.clone(), step.loss.item(), step.turn_sum.clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    assert outs[0][2] == outs[1][2] and torch.equal(outs[0][3], outs[1][3])


def test_device_errors(P, oracle):
    b = W.tiny()
    V = 64
    zs, zt = W.make_logits(b.num_tokens, V, "tiny", torch.float32, seed=0, device="cuda")
    valid = np.nonzero(b.loss_mask)[0]
    # row index out of range -> TOKEN_RANGE, that token's loss is 0, the rest unaffected
    step = make_step(P, b, V, compact=True)
    step.row_of_token[int(valid[5])] = b.num_valid + 3
    step.run(zs[:b.num_valid], zt[:b.num_valid], torch.zeros_like(zs[:b.num_valid]))
    torch.cuda.synchronize()
    assert step.status() == 5
    assert step.token_loss[int(valid[5])].item() == 0.0
    # sampled id out of range
    y = torch.zeros(b.num_tokens, dtype=torch.int32, device="cuda")
    y[int(valid[2])] = V
    step = make_step(P, b, V, compact=False, mode=1, y=y)
    step.run(zs, zt, torch.zeros_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 5
    # supervised token with a turn id out of range
    step = make_step(P, b, V, compact=False)
    step.turn_id[int(valid[0])] = b.max_turns
    step.run(zs, zt, torch.zeros_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 4
    # bad offsets
    step = make_step(P, b, V, compact=False)
    step.traj_offsets[1] = b.num_tokens + 5
    step.weights()
    torch.cuda.synchronize()
    assert step.status() == 3
    # non-finite logits
    step = make_step(P, b, V, compact=False)
    zs2 = zs.clone()
    zs2[int(valid[1]), 3] = float("inf")
    step.run(zs2, zt, torch.zeros_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 9


def test_virtual_ranks_merge(P, oracle):
    """Data-parallel by whole trajectories, emulated on one GPU: each 'rank' runs its
    own trajectories with the rank-summed count vector; merged results equal one call."""
    b = W.packed(seed=9, num_traj=6, traj_len=1024)
    V = 3000
    zs, zt = W.make_logits(b.num_tokens, V, "agent", torch.bfloat16, seed=9, device="cuda")
    whole = make_step(P, b, V, compact=False, alpha=0.6, scope=0, n_min=2)
    gw = torch.zeros_like(zs)
    whole.run(zs, zt, gw)
    parts, steps = [(0, 2), (2, 6)], []
    for lo, hi in parts:
        a, z = int(b.traj_offsets[lo]), int(b.traj_offsets[hi])
        sub = W.Batch("part", b.turn_id[a:z], b.loss_mask[a:z], b.traj_offsets[lo:hi + 1] - a,
                      b.max_turns)
        steps.append((make_step(P, sub, V, compact=False, alpha=0.6, scope=0, n_min=2), a, z))
    g_counts = sum(s.local_counts().clone() for s, _, _ in steps)
    grads = []
    for s, a, z in steps:
        g = torch.zeros_like(zs[a:z])
        s.run(zs[a:z], zt[a:z], g, global_counts=g_counts)
        grads.append(g)
    torch.cuda.synchronize()
    assert whole.status() == 0 and all(s.status() == 0 for s, _, _ in steps)
    assert torch.equal(torch.cat([s.w[:s.T] for s, _, _ in steps]), whole.w[:whole.T])
    assert torch.equal(torch.cat(grads), gw)
    loss = sum(s.loss.item() for s, _, _ in steps)
    assert abs(loss - whole.loss.item()) <= 1e-12 * abs(whole.loss.item())
    assert torch.equal(sum(s.turn_cnt for s, _, _ in steps), whole.turn_cnt)
    assert torch.equal(sum(s.turn_surv for s, _, _ in steps), whole.turn_surv)
    torch.testing.assert_close(sum(s.turn_sum for s, _, _ in steps), whole.turn_sum,
                               rtol=1e-12, atol=1e-12)
