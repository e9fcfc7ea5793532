"""One loss step captured in a CUDA graph and replayed gives the same bits as the
stream-ordered call (weights, both row grids with the helper's programmatic launch
-- or, for fp32 logits, the split-row kernel's clusters -- the loss sum and the
turn statistics)."""
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("mode", [0, 1], ids=["full", "sampled"])
def test_step_in_a_cuda_graph_matches_eager(mode, dtype):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P
    from paper_2607_05804_gb300.step import LossStep, to_device

    P.load()
    b = W.packed(seed=5, num_traj=2, traj_len=1024)
    V = W.V_QWEN
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16 if dtype == "bf16" else torch.float32,
                           seed=5, device="cuda")
    tid, msk, off, rot = to_device(b, "cuda", compact=True)
    y = None
    if mode == 1:
        y_rows = W.sample_ids(zs, 6)
        y = torch.zeros(b.num_tokens, dtype=torch.int32, device="cuda")
        y[torch.from_numpy(b.loss_mask.nonzero()[0]).cuda()] = y_rows
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, sampled_ids=y, mode=mode, alpha=0.5)
    grad = torch.empty_like(zs)
    step.run(zs, zt, grad)
    torch.cuda.synchronize()
    assert step.status() == 0
    ref = (step.loss.clone(), step.token_loss.clone(), grad.clone(), step.turn_sum.clone())

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step.run(zs, zt, grad)  # warm-up on the capture stream
    torch.cuda.current_stream().wait_stream(side)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step.run(zs, zt, grad)
    grad.zero_()
    step.loss.zero_()
    step.token_loss.zero_()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert step.status() == 0
    assert torch.equal(step.loss, ref[0])
    assert torch.equal(step.token_loss, ref[1])
    assert torch.equal(grad, ref[2])
    assert torch.equal(step.turn_sum, ref[3])
