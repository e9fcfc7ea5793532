"""The no-allocation loss entry point (turnopd_loss_fwd_bwd_static) against the
workspace entry point (turnopd_loss_fwd_bwd).

turnopd_loss_fwd_bwd_static exists for callers that cannot allocate device
memory (their memory belongs to an allocator or arena that forbids raw
cudaMalloc/cudaFree, or they have no allocator to hand out a workspace); it keeps
its scratch in a static device array inside the library.  Three calls in a row,
with different inputs and sizes, must each match the workspace entry point on
the same inputs bit for bit (the library's outputs are bitwise reproducible),
so nothing left in the shared array by one call leaks into the next; and they
must leave the device's free memory unchanged.  This file is collected last on
purpose.
"""
import numpy as np
import pytest

import workloads as W

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
    """Three static calls in a row (a large batch, a smaller one with another vocabulary
    and mode, then the large one again, so a leftover of either call in the shared
    array would show), each against the workspace entry point on the same inputs.
    After one warm-up call of each case, the static calls change neither the device's
    free memory nor torch's allocated bytes."""
    cases = [(W.packed(seed=21, num_traj=2, traj_len=4096), W.V_QWEN, 21, 0),
             (W.household(seed=22, num_traj=2, traj_len=2048), 50000, 22, 1)]
    prepared = []
    for b, V, seed, mode in cases:
        assert b.num_tokens <= P.TURNOPD_STATIC_MAX_TOKENS
        zs, zt, msk, rot, w, y = _inputs(b, V, seed, mode)
        T = b.num_tokens
        ws = torch.empty(P.turnopd_loss_workspace_bytes(T), dtype=torch.uint8, device="cuda")
        ref = _outputs(zs, T)
        g_ref, tl_ref, l_ref, st_ref = ref
        P.turnopd_loss_fwd_bwd(zs, zt, V, rot, y, msk, w, mode, g_ref, 0, tl_ref, l_ref, ws, st_ref)
        prepared.append((b, V, mode, (zs, zt, msk, rot, w, y), ref))
    order = [0, 1, 0]
    outs = [_outputs(prepared[c][3][0], prepared[c][0].num_tokens) for c in order]

    def call(case, out):
        b, V, mode, (zs, zt, msk, rot, w, y), _ = prepared[case]
        g, tl, l, st = out
        P.turnopd_loss_fwd_bwd_static(zs, zt, V, rot, y, msk, w, mode, g, 0, tl, l, st)

    for c in range(len(cases)):   # warm-up: kernels of both cases loaded on the device
        call(c, _outputs(prepared[c][3][0], prepared[c][0].num_tokens))
    torch.cuda.synchronize()
    free0, alloc0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_allocated()
    for c, out in zip(order, outs):
        call(c, out)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.cuda.memory_allocated() == alloc0

    for c, (g, tl, l, st) in zip(order, outs):
        b, V, mode, (zs, zt, msk, rot, w, y), (g_ref, tl_ref, l_ref, st_ref) = prepared[c]
        assert st_ref.item() == 0 and st.item() == 0
        # the same kernels on the same inputs: the library's results are bitwise
        # reproducible, so only the scratch's home differs
        assert torch.equal(tl, tl_ref) and torch.equal(l, l_ref) and torch.equal(g, g_ref)


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
