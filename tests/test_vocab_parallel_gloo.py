"""World-size-2 gloo test of the vocabulary-parallel exchange (CPU only).

Each rank holds one column shard of the logits, reduces it to partial row
statistics (oracle), all-gathers the partials in rank order, merges them and
writes its gradient columns.  The gathered result must equal the
full-vocabulary oracle: the per-token loss on every rank, and the gradient
columns concatenated in rank order."""
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")

R, V, CUT = 20, 333, 149   # uneven shards


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _data():
    rng = np.random.default_rng(5)
    zs = rng.normal(0, 3, (R, V)).astype(np.float32).astype(np.float64)   # float32-exact values
    zt = (0.8 * zs + rng.normal(0, 2, (R, V))).astype(np.float32).astype(np.float64)
    w = rng.random(R)
    return zs, zt, w


def _rank_main(rank, world, port, result_path):
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import torch.distributed as dist

    from oracle import vocab_parallel as VP

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    zs, zt, w = _data()
    lo, hi = (0, CUT) if rank == 0 else (CUT, V)
    part = torch.from_numpy(VP.shard_stats(zs[:, lo:hi], zt[:, lo:hi]))
    parts = [torch.empty_like(part) for _ in range(world)]
    dist.all_gather(parts, part)
    merged = VP.merge(torch.stack(parts).numpy())
    kl = VP.row_constants(merged)[3]
    g = torch.from_numpy(VP.shard_grad(zs[:, lo:hi], zt[:, lo:hi], merged, w))
    sizes = [CUT, V - CUT]
    gs = [torch.empty((R, n), dtype=torch.float64) for n in sizes]
    if rank == 0:
        gs[0] = g
        dist.recv(gs[1], src=1)
    else:
        dist.send(g, dst=0)
    kls = [torch.empty(R, dtype=torch.float64) for _ in range(world)]
    dist.all_gather(kls, torch.from_numpy(kl))
    if rank == 0:
        import pickle

        with open(result_path, "wb") as fh:
            pickle.dump((torch.cat(gs, dim=1).numpy(), [k.numpy() for k in kls]), fh)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_vocab_split_equals_full_vocabulary(oracle, tmp_path):
    import pickle

    import torch.multiprocessing as mp

    port = _free_port()
    path = str(tmp_path / "res.pkl")
    mp.spawn(_rank_main, args=(2, port, path), nprocs=2, join=True)
    with open(path, "rb") as fh:
        g, kls = pickle.load(fh)
    zs, zt, w = _data()
    assert np.array_equal(kls[0], kls[1])          # every rank holds the same row constants
    for r in range(R):
        _, _, _, kl, gr = oracle.row(zs[r].astype(np.float32), zt[r].astype(np.float32), w=float(w[r]))
        assert abs(kls[0][r] - kl) <= 1e-12 * max(1.0, kl)
        np.testing.assert_allclose(g[r], gr, rtol=0, atol=1e-14 * np.abs(gr).max())
