"""The rollout-depth controller fed with the per-turn tables of a real loss
step on the GPU (the tables are copied to the host), against the controller
oracle on the same tables."""
import numpy as np
import pytest

import workloads as W
from oracle import controller as C

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def test_controller_on_gpu_turn_stats():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2607_05804_gb300 as P
    from paper_2607_05804_gb300.controller import DepthController
    from paper_2607_05804_gb300.step import LossStep, to_device

    P.load()
    b = W.household(seed=2)
    V = 4096
    zs, zt = W.make_logits(b.num_valid, V, "agent", torch.bfloat16, seed=21, device="cuda")
    tid, msk, off, rot = to_device(b, "cuda", compact=True)
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, alpha=0.5)
    step.run(zs, zt, torch.empty_like(zs))
    torch.cuda.synchronize()
    assert step.status() == 0
    # trajectory length = turns that hold a supervised token; success drawn at random
    lens = np.array([len(set(b.turn_id[b.traj_offsets[i]:b.traj_offsets[i + 1]][
        b.loss_mask[b.traj_offsets[i]:b.traj_offsets[i + 1]] == 1].tolist())) for i in range(b.num_traj)])
    succ = np.random.default_rng(0).random(b.num_traj) < 0.6
    ctl = DepthController(min_cov_traj=4)
    ref = C.Controller(min_cov_traj=4)
    for k in (1, 2, 3):
        assert ctl.plan(k) == ref.plan(k)
        ctl.update(k, step, lens, succ)
        ref.update(k, step.turn_sum.cpu().numpy(), step.turn_cnt.cpu().numpy(), step.turn_surv.cpu().numpy(),
                   lens, succ)
        assert ctl.state.h_bar == ref.hbar and ctl.state.h_cov == ref.h_cov and ctl.state.h_eff == ref.h_eff
    bsh, ssh, deep = DepthController.diagnostics(step, n_min=2)
    d = C.diagnostics(step.turn_sum.cpu().numpy(), step.turn_cnt.cpu().numpy(), step.turn_surv.cpu().numpy(), 2)
    np.testing.assert_allclose(ssh, d["s"], rtol=1e-12, atol=1e-15)
    assert deep[0] == d["prefix"]
