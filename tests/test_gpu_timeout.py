"""The device-side timeout path: a bounded wait that runs out records
TURNOPD_ERR_TIMEOUT and returns, and the stream stays usable.  The wait is on a
barrier that nothing arrives on (no failure of the GPU is involved)."""
import numpy as np
import pytest

import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TURNOPD_ERR_TIMEOUT = 8


def test_wait_timeout_is_reported_and_the_stream_stays_usable():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import oracle
    import paper_2607_05804_gb300 as P
    from paper_2607_05804_gb300.step import LossStep, to_device

    P.load()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    for limit in (1, 1000, 1 << 16):
        st.zero_()
        P.turnopd_selftest_wait_timeout(limit, st)
        torch.cuda.synchronize()
        assert int(st.item()) == TURNOPD_ERR_TIMEOUT
    # a loss step on the same stream afterwards is unaffected
    b = W.packed(seed=3, num_traj=2, traj_len=128)
    V = 1000
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=3, device="cuda")
    tid, msk, off, rot = to_device(b, "cuda", compact=True)
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, alpha=0.5)
    step.run(zs, zt, torch.empty_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 0
    oracle.build()
    w = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, 0.5)
    _, _, loss_ref = oracle.loss_fwd_bwd(W.bf16_bits(zs), W.bf16_bits(zt), V, b.loss_mask,
                                         w.astype(np.float32), row_of_token=b.compact_rows(), grad=False)
    assert abs(step.loss.item() - loss_ref) <= 1e-5 * abs(loss_ref)
