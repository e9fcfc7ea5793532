"""World-size-2 gloo test of the data-parallel host logic (CPU only).

Each rank owns half of the trajectories of one batch, computes its count vector
and weights with the fp64 oracle, sums the count vectors through
paper_2607_05804_gb300.dp.global_counts, and reduces loss and turn statistics
through dp.reduce_step, which packs them into one all-reduce.  The merged results must equal the single-process oracle
on the whole batch: weights and counts exactly, sums within fp64 rounding."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, result_path):
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch.distributed as dist

    import oracle
    import workloads as W
    from paper_2607_05804_gb300 import dp

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = W.packed(seed=3, num_traj=6, traj_len=256)
    cut = [0, 2, 6]
    lo, hi = cut[rank], cut[rank + 1]
    a, z = int(b.traj_offsets[lo]), int(b.traj_offsets[hi])
    tid, msk = b.turn_id[a:z], b.loss_mask[a:z]
    off = b.traj_offsets[lo:hi + 1] - a
    V = 64
    rng = np.random.default_rng(0)
    zs_all = rng.normal(0, 3, (b.num_tokens, V)).astype(np.float32)
    zt_all = (0.8 * zs_all + rng.normal(0, 2, (b.num_tokens, V))).astype(np.float32)
    zs, zt = zs_all[a:z], zt_all[a:z]
    out = {}
    for scope, n_min in ((0, 0), (0, 2), (1, 0), (1, 3)):
        _, local = oracle.turn_counts(tid, msk, off, b.max_turns)
        g = dp.global_counts(torch.from_numpy(local)).numpy()
        w = oracle.weights(tid, msk, off, b.max_turns, 0.4, scope, n_min, global_counts=g)
        _, tl, loss = oracle.loss_fwd_bwd(zs, zt, V, msk, w.astype(np.float32))
        st = oracle.turn_stats(tl, tid, msk, off, b.max_turns)
        L = torch.tensor([loss], dtype=torch.float64)
        ts = torch.from_numpy(st["turn_sum"].copy())
        tc = torch.from_numpy(st["turn_cnt"].copy())
        sv = torch.from_numpy(st["turn_surv"].copy())
        calls = []
        real = dist.all_reduce
        dist.all_reduce = lambda *a, **k: (calls.append(1), real(*a, **k))[1]
        try:
            dp.reduce_step(L, ts, tc, sv)
        finally:
            dist.all_reduce = real
        assert len(calls) == 1  # one packed collective after the step
        assert tc.dtype == torch.int64 and sv.dtype == torch.int32
        parts = [None] * world
        dist.all_gather_object(parts, w)
        out[(scope, n_min)] = (np.concatenate(parts), L.item(), ts.numpy(), tc.numpy(), sv.numpy())
    if rank == 0:
        import pickle

        with open(result_path, "wb") as fh:
            pickle.dump(out, fh)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_merge_equals_single_batch(oracle, tmp_path):
    import pickle

    import torch.multiprocessing as mp

    import workloads as W

    port = _free_port()
    path = str(tmp_path / "res.pkl")
    mp.spawn(_rank_main, args=(2, port, path), nprocs=2, join=True)
    with open(path, "rb") as fh:
        res = pickle.load(fh)
    b = W.packed(seed=3, num_traj=6, traj_len=256)
    V = 64
    rng = np.random.default_rng(0)
    zs = rng.normal(0, 3, (b.num_tokens, V)).astype(np.float32)
    zt = (0.8 * zs + rng.normal(0, 2, (b.num_tokens, V))).astype(np.float32)
    for (scope, n_min), (w, loss, ts, tc, sv) in res.items():
        w_ref = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, 0.4, scope, n_min)
        assert np.array_equal(w, w_ref)
        _, tl, loss_ref = oracle.loss_fwd_bwd(zs, zt, V, b.loss_mask, w_ref.astype(np.float32))
        st = oracle.turn_stats(tl, b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns)
        assert abs(loss - loss_ref) <= 1e-12 * abs(loss_ref)
        np.testing.assert_allclose(ts, st["turn_sum"], rtol=1e-12, atol=1e-12)
        assert np.array_equal(tc, st["turn_cnt"]) and np.array_equal(sv, st["turn_surv"])
