"""The no-allocation loss entry point (turnopd_loss_fwd_bwd_static) against the
workspace entry point (turnopd_loss_fwd_bwd).

turnopd_loss_fwd_bwd_static exists for callers that cannot allocate device
memory (their memory belongs to an allocator or arena that forbids raw
cudaMalloc/cudaFree, or they have no allocator to hand out a workspace); it keeps
its scratch in a static device array inside the library.  Two calls in a row,
with different inputs and sizes, must each match the workspace entry point on
the same inputs within the parity tolerances, so nothing left in the shared
array by one call leaks into the next.  This file is collected last on purpose.
"""
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


def _inputs(b, V, seed, mode):
    from paper_2607_05804_gb300.step import to_device

    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=seed, device="cuda")
    tid, msk, off, rot = to_device(b, "cuda", compact=True)
    rng = np.random.default_rng(seed)
    w = torch.from_numpy((rng.random(b.num_tokens) * b.loss_mask).astype(np.float32)).cuda()
    y = None
    if mode == 1:
        y = torch.zeros(b.num_tokens, dtype=torch.int32, device="cuda")
        y[torch.from_numpy(np.nonzero(b.loss_mask)[0]).cuda()] = W.sample_ids(zs, seed + 7)
    return zs, zt, msk, rot, w, y


def _outputs(zs, T):
    return (torch.zeros_like(zs), torch.zeros(T, dtype=torch.float32, device="cuda"),
            torch.zeros(1, dtype=torch.float64, device="cuda"),
            torch.zeros(1, dtype=torch.int32, device="cuda"))


def test_static_entry_matches_workspace_entry_twice(P):
    cases = [(W.packed(seed=21, num_traj=2, traj_len=4096), W.V_QWEN, 21, 0),
             (W.household(seed=22, num_traj=2, traj_len=2048), 50000, 22, 1)]
    for b, V, seed, mode in cases:  # two calls in a row, second one smaller and different
        assert b.num_tokens <= P.TURNOPD_STATIC_MAX_TOKENS
        zs, zt, msk, rot, w, y = _inputs(b, V, seed, mode)
        T = b.num_tokens
        ws = torch.empty(P.turnopd_loss_workspace_bytes(T), dtype=torch.uint8, device="cuda")
        g_ref, tl_ref, l_ref, st_ref = _outputs(zs, T)
        P.turnopd_loss_fwd_bwd(zs, zt, V, rot, y, msk, w, mode, g_ref, 0, tl_ref, l_ref, ws, st_ref)
        g, tl, l, st = _outputs(zs, T)
        P.turnopd_loss_fwd_bwd_static(zs, zt, V, rot, y, msk, w, mode, g, 0, tl, l, st)
        torch.cuda.synchronize()
        assert st_ref.item() == 0 and st.item() == 0
        tl_ref_np = tl_ref.cpu().numpy().astype(np.float64)
        assert_token_loss(tl.cpu().numpy(), tl_ref_np, b.loss_mask)
        assert_loss(l.item(), l_ref.item())
        rows = np.arange(0, b.num_valid, max(1, b.num_valid // 64))
        toks = np.nonzero(b.loss_mask)[0][rows]
        extra = dict(ell=tl_ref_np[toks], w=w.cpu().numpy()[toks]) if mode == 1 else {}
        assert_grad_rows(g[rows].float().cpu().numpy(), g_ref[rows].float().cpu().numpy(),
                         bf16=True, **extra)


def test_static_entry_rejects_oversized_batches(P):
    T = P.TURNOPD_STATIC_MAX_TOKENS + 1
    z = torch.zeros((1, 8), dtype=torch.bfloat16, device="cuda")
    msk = torch.zeros(T, dtype=torch.uint8, device="cuda")
    rot = torch.full((T,), -1, dtype=torch.int32, device="cuda")
    w = torch.zeros(T, dtype=torch.float32, device="cuda")
    tl = torch.zeros(T, dtype=torch.float32, device="cuda")
    loss = torch.zeros(1, dtype=torch.float64, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    with pytest.raises(P.TurnopdError) as e:
        P.turnopd_loss_fwd_bwd_static(z, z, 8, rot, None, msk, w, 0, None, 0, tl, loss, st)
    assert e.value.code == 10
