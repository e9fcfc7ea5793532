#!/usr/bin/env python3
"""Benchmark of the turn-aware OPD loss step on GB300.

A step is one pass of the whole hot path over one packed batch: blend weights
(turnopd_weights), per-token reverse KL + student-logit gradient + weighted
loss (turnopd_loss_fwd_bwd) and turn statistics (turnopd_turn_stats).

Default workload: 8 trajectories x 4096 tokens, 10-30 turns, 40 % masked
observation tokens, V = 151,936, bf16 logits (compact rows: one per supervised
token), bf16 gradient, alpha = 0.5, full-vocabulary mode.  Inputs are seeded
synthetic data already resident in HBM; each step streams ~17.9 GB, far more
than the 129 MB L2, so no flush is needed between steps.

Prints one JSON line (rank 0).  --impl reference times the fp64 CPU oracle on a
bounded sample of the same workload instead.

Under torchrun with N > 1 every rank runs its own batch (weak scaling); the
ranks exchange the count vector before the weights and the loss after the step
(NCCL all-reduce of 2*max_turns+2 numbers), the path's only cross-rank data.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "loss fwd+bwd tokens/s at V=151936 bf16 on 1 GB300; achieved HBM GB/s vs peak"
UNIT = "tokens/s"
V_QWEN = 151_936  # the workloads' vocabulary (a --vocab run has no committed traffic record)
# counts(2) + weights(1) + compaction(2) + row kernel + loss sum + stats(2); the full and
# sampled modes add the helper grid that runs beside the cluster grid (k_row_helper for
# bf16 logits, k_split_helper for fp32)
KERNELS_PER_STEP = 9
ROW_KERNEL_SOURCES = ["paper_2607_05804_gb300/csrc/rowkl_cluster.cuh",
                      "paper_2607_05804_gb300/csrc/rowkl_cluster.cu",
                      "paper_2607_05804_gb300/csrc/loss_kernels.cu",
                      "paper_2607_05804_gb300/csrc/common.cuh",
                      "paper_2607_05804_gb300/csrc/row_math.cuh",
                      "paper_2607_05804_gb300/csrc/packed.cuh"]


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["native", "reference"], default="native")
    p.add_argument("--workload", default="packed", choices=["packed", "household", "multihop", "fused"])
    p.add_argument("--mode", default="full", choices=["full", "sampled", "topk"])
    p.add_argument("--k-top", type=int, default=50, help="support size of --mode topk")
    p.add_argument("--dw", action="store_true", help="fused workload: also the weight gradient dL/dW_s")
    p.add_argument("--vocab-shards", type=int, default=0,
                   help="time the vocabulary-parallel path with this many column shards of one GPU's logits "
                        "standing in for ranks (stats, ordered merge, shard gradients)")
    p.add_argument("--layout", default="compact", choices=["compact", "dense"],
                   help="logit rows: one per supervised token, or one per token (row i = token i)")
    p.add_argument("--zero-masked", action="store_true",
                   help="dense layout with TURNOPD_ZERO_MASKED_GRAD: masked tokens' gradient rows written as zeros")
    p.add_argument("--fp32-grad", action="store_true", help="full/sampled modes: an fp32 gradient instead of bf16")
    p.add_argument("--vocab", type=int, default=0,
                   help="full/sampled/top-K modes: vocabulary size (0 = the workload's 151,936)")
    p.add_argument("--fp32-logits", action="store_true",
                   help="full/sampled modes: fp32 logits instead of bf16 (the split-row kernel)")
    p.add_argument("--alpha", type=float, default=0.5)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-sample-rows", type=int, default=0, help="0 = size to ~15 s of oracle work")
    p.add_argument("--num-traj", type=int, default=0,
                   help="packed and fused workloads: trajectories (0 = 8); smaller cases serve profiling")
    p.add_argument("--traj-len", type=int, default=0, help="packed and fused workloads: tokens per trajectory (0 = the workload's own)")
    return p.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


TOPK_KERNEL_SOURCES = ["paper_2607_05804_gb300/csrc/topk_kernels.cu",
                       "paper_2607_05804_gb300/csrc/common.cuh"]


def source_hash(sources=None):
    h = hashlib.sha256()
    for rel in (ROW_KERNEL_SOURCES if sources is None else sources):
        with open(os.path.join(ROOT, rel), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def committed_traffic(workload, rows=None, kind="row"):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on the
    current kernel source: the row kernels' per-workload figure, or (kind "topk")
    the top-K kernel's bytes per row times `rows`."""
    name, sources = (("topk_traffic.json", TOPK_KERNEL_SOURCES) if kind == "topk"
                     else ("row_kernel_traffic.json", ROW_KERNEL_SOURCES))
    try:
        with open(os.path.join(ROOT, "profiles", name)) as fh:
            d = json.load(fh)
        if d.get("source_hash") != source_hash(sources):
            return None
        if kind == "topk":
            return d["bytes_per_row"] * rows
        return d.get("bytes_per_launch", {}).get(workload)
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index, self.rows, self.proc = index, [], None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 8:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.thread.join(timeout=2)
        if not self.rows:
            return None
        sm = [float(r[0]) for r in self.rows if r[0].replace(".", "").isdigit()]
        mx = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in self.rows for k in range(4) if r[4 + k] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(self.rows)}


def dense_layout(args):
    return args.layout == "dense" or args.zero_masked


def build_inputs(args, rank, device):
    import torch

    import workloads as W
    from paper_2607_05804_gb300 import TURNOPD_FULL_VOCAB, TURNOPD_SAMPLED_TOKEN
    from paper_2607_05804_gb300.step import LossStep, to_device

    if args.workload == "packed" and (args.num_traj or args.traj_len):
        b = W.packed(seed=rank, num_traj=args.num_traj or 8, traj_len=args.traj_len or 4096)
    else:
        b = W.CONFIGS[args.workload](seed=rank)
    from paper_2607_05804_gb300 import TURNOPD_ZERO_MASKED_GRAD

    V = args.vocab or W.V_QWEN
    dense = dense_layout(args)
    rows = b.num_tokens if dense else b.num_valid
    zs, zt = W.make_logits(rows, V, "agent", torch.float32 if args.fp32_logits else torch.bfloat16,
                           seed=1000 + rank, device=device)
    mode = TURNOPD_SAMPLED_TOKEN if args.mode == "sampled" else TURNOPD_FULL_VOCAB
    y = None
    if mode == TURNOPD_SAMPLED_TOKEN:
        y_c = W.sample_ids(zs, seed=2000 + rank)  # per row; expand to per token
        if dense:
            y = y_c
        else:
            y = torch.zeros(b.num_tokens, dtype=torch.int32, device=device)
            idx = torch.from_numpy(b.loss_mask.nonzero()[0]).to(device)
            y[idx] = y_c
    tid, msk, off, rot = to_device(b, device, compact=not dense)
    k_top = args.k_top if args.mode == "topk" else 0
    step = LossStep(tid, msk, off, b.max_turns, V, row_of_token=rot, sampled_ids=y, mode=mode,
                    alpha=args.alpha, k_top=k_top, flags=TURNOPD_ZERO_MASKED_GRAD if args.zero_masked else 0)
    # the top-K mode returns its gradient sparse: (ids, values) per token
    grad = None if k_top else torch.empty(zs.shape, dtype=torch.float32 if args.fp32_grad else zs.dtype,
                                          device=zs.device)
    return b, V, zs, zt, grad, step


def vocab_parallel_loss_fn(step, zs, zt, grad, n_shards):
    """One loss call of the vocabulary-parallel path with n_shards column shards of
    this GPU's logits: every shard's statistics, the ordered merge, every shard's
    gradient columns (the work all ranks of an n_shards-way split do together)."""
    import torch

    import paper_2607_05804_gb300 as P

    V = step.vocab
    T = step.T
    cuts = [V * r // n_shards for r in range(n_shards + 1)]
    if not hasattr(step, "_vp"):
        step._vp = (torch.empty((n_shards, T, 6), dtype=torch.float32, device=zs.device),
                    torch.empty((T, 6), dtype=torch.float32, device=zs.device))
    parts, merged = step._vp

    def call():
        for r in range(n_shards):
            P.turnopd_vocab_shard_stats(zs[:, cuts[r]:cuts[r + 1]], zt[:, cuts[r]:cuts[r + 1]], step.row_of_token,
                                        step.loss_mask, parts[r], step.ws_l, step.dev_status)
        P.turnopd_vocab_stats_merge(parts, step.loss_mask, merged)
        for r in range(n_shards):
            P.turnopd_vocab_shard_loss_grad(zs[:, cuts[r]:cuts[r + 1]], zt[:, cuts[r]:cuts[r + 1]],
                                            step.row_of_token, step.loss_mask, step.w[:T], merged,
                                            grad[:, cuts[r]:cuts[r + 1]], 0, step.token_loss[:T], step.loss,
                                            step.ws_l, step.dev_status)
    return call


def run_step(step, zs, zt, grad, world, dist, ev_pair=None):
    from paper_2607_05804_gb300 import dp

    if world > 1:
        step.weights(dp.global_counts(step.local_counts()))
    else:
        step.weights()
    if ev_pair is not None:
        ev_pair[0].record()
    if getattr(step, "vp_call", None) is not None:
        step.vp_call()
    else:
        step.loss_fwd_bwd(zs, zt, grad)
    if ev_pair is not None:
        ev_pair[1].record()
    step.turn_stats()
    if world > 1:
        dp.reduce_step(step.loss, step.turn_sum, step.turn_cnt, step.turn_surv)


def cpu_baseline(b, zs, zt, V, alpha, mode, rows_override=0, budget_s=15.0, k_top=0, dense=False):
    """Time the fp64 CPU oracle on a bounded sample of the same workload: supervised
    rows in order, in chunks of 512 (so the oracle's fp64 gradient stays a few GB),
    until about `budget_s` seconds of oracle time or `rows_override` rows."""
    import numpy as np
    import torch

    import oracle
    import workloads as W

    oracle.build()
    w = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, alpha).astype(np.float32)
    valid = np.nonzero(b.loss_mask)[0]
    R = valid.size
    limit = min(R, rows_override) if rows_override else R
    done, spent, chunk = 0, 0.0, 512
    while done < limit and (rows_override or spent < budget_s):
        n = min(chunk, limit - done)
        host = W.bf16_bits if zs.dtype == torch.bfloat16 else (lambda t: t.cpu().numpy())
        if dense:  # the supervised tokens' own rows
            sel = torch.from_numpy(valid[done:done + n]).to(zs.device)
            zsn, ztn = host(zs.index_select(0, sel)), host(zt.index_select(0, sel))
        else:
            zsn, ztn = host(zs[done:done + n]), host(zt[done:done + n])
        t0 = time.perf_counter()
        if k_top:
            oracle.topk_loss(zsn, ztn, V, np.ones(n, np.uint8), w[valid[done:done + n]], k_top)
        else:
            oracle.loss_fwd_bwd(zsn, ztn, V, np.ones(n, np.uint8), w[valid[done:done + n]], mode=0)
        spent += time.perf_counter() - t0
        done += n
    what = (f"teacher top-{k_top} reverse KL and its sparse gradient" if k_top
            else "full-vocabulary loss and gradient")
    return {"value": done / spent, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"first {done} supervised rows of the same batch, {what} in fp64 "
                      f"({spent:.1f} s of oracle time, chunks of {chunk} rows)"}


def reference_arm(args, world, rank):
    """--impl reference: the fp64 CPU oracle as the reference implementation."""
    import numpy as np

    import oracle
    import workloads as W

    if rank != 0:
        return
    import torch

    b = W.CONFIGS[args.workload](seed=0)
    V = W.V_QWEN
    n = 32  # rows per reference step (bounded so the whole run ends within minutes)
    zs, zt = W.make_logits(n, V, "agent", torch.bfloat16, seed=1000, device="cpu", chunk_rows=8)
    zsb, ztb = W.bf16_bits(zs), W.bf16_bits(zt)
    w = oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, args.alpha)
    valid = np.nonzero(b.loss_mask)[0]
    w32 = w.astype(np.float32)[valid[:n]]
    mask = np.ones(n, np.uint8)
    times = []
    for k in range(args.warmup + args.steps):
        t0 = time.perf_counter()
        oracle.weights(b.turn_id, b.loss_mask, b.traj_offsets, b.max_turns, args.alpha)
        _, tl, _ = oracle.loss_fwd_bwd(zsb, ztb, V, mask, w32, mode=0)
        dt = time.perf_counter() - t0
        if k >= args.warmup:
            times.append(dt)
    tot = sum(times)
    value = n * len(times) / tot
    cores = oracle.num_threads()
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": 1e3 * tot / len(times), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "impl": "reference",
           "config": {"workload": f"{b.name}_V{V}", "sample_rows_per_step": n},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                            "sample": f"{n} supervised rows per step of the {b.name} batch"},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# weights (3) + fused call (compaction 2, gathers 2, statistics pass, merge, gradient
# pass, masked-row zeroing, dL/dh_s, dL/dh_s fix-up, loss sum) + turn statistics (2)
FUSED_KERNELS_PER_STEP = 16


def fused_cpu_baseline(b, heads, w, budget_s=12.0):
    """The fp64 oracle on a bounded sample of supervised tokens of the fused
    workload (each token: both heads' logits over the whole vocabulary, the KL,
    and dL/dh_s), scaled to supervised tokens/s."""
    import numpy as np

    import oracle
    import workloads as W

    bits = [W.bf16_bits(x) for x in heads]
    wn = w.cpu().numpy()
    valid = np.nonzero(b.loss_mask)[0]
    n, spent = 4, 0.0
    while True:
        pick = valid[:: max(1, len(valid) // n)][:n]
        t0 = time.perf_counter()
        oracle.fused_lmhead(*bits, b.loss_mask, wn, subset=pick)
        spent = time.perf_counter() - t0
        if spent > budget_s / 4 or n >= len(valid):
            break
        n = min(len(valid), int(n * max(2.0, budget_s / 2 / max(spent, 1e-3))))
    return {"value": len(pick) / spent, "unit": "tokens/s", "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{len(pick)} of {len(valid)} supervised tokens, full heads, fp64, {spent:.1f} s"}


def fused_bench(args, world, rank, local):
    """Fused LM-head step: 8 x 2048 tokens (packed turn structure), student head
    4096 x 151,936, teacher head 5120 x 151,936 (bf16), alpha = 1, full vocabulary:
    weights, fused forward + backward (dL/dh_s), turn statistics."""
    import torch

    import workloads as W
    import paper_2607_05804_gb300 as P
    from paper_2607_05804_gb300.step import LossStep, to_device

    from paper_2607_05804_gb300 import dp

    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    dist = None
    if world > 1:
        import torch.distributed as dist

        dist.init_process_group("nccl", device_id=device)
    P.load()
    b = W.fused(seed=rank, num_traj=args.num_traj or 8, traj_len=args.traj_len or 2048)
    d_s, d_t, V = 4096, 5120, W.V_QWEN
    T = b.num_tokens
    h_s, W_s, h_t, W_t = W.make_fused(T, d_s, d_t, V, seed=3000 + rank, device=device)
    tid, msk, off, _ = to_device(b, device, compact=False)
    step = LossStep(tid, msk, off, b.max_turns, V, alpha=1.0)
    ws = torch.empty(P.turnopd_fused_workspace_bytes(T, V, d_s, d_t), dtype=torch.uint8, device=device)
    dh = torch.empty((T, d_s), dtype=torch.float32, device=device)
    dW = torch.empty((V, d_s), dtype=torch.float32, device=device) if args.dw else None

    def one(ev=None):
        step.weights(dp.global_counts(step.local_counts()) if world > 1 else None)
        if ev is not None:
            ev[0].record()
        P.turnopd_fused_lmhead_fwd_bwd(h_s, W_s, h_t, W_t, msk, step.w[:T], 0, dh,
                                       step.token_loss[:T], step.loss, ws, step.dev_status, dW_s_out=dW)
        if ev is not None:
            ev[1].record()
        step.turn_stats()
        if world > 1:
            dp.reduce_step(step.loss, step.turn_sum, step.turn_cnt, step.turn_surv)

    for _ in range(max(args.warmup, 3)):
        one()
    torch.cuda.synchronize()
    if step.status() != 0:
        raise RuntimeError(f"device status {step.status()}")
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    a.record()
    for k in range(args.steps):
        one(evs[k])
    z.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms = a.elapsed_time(z)
    call_ms = statistics.mean(x.elapsed_time(y) for x, y in evs)
    Tv = b.num_valid
    tot_valid = Tv
    if world > 1:
        t = torch.tensor([ms, call_ms], device=device, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms, call_ms = float(t[0].item()), float(t[1].item())
        n = torch.tensor([Tv], device=device, dtype=torch.int64)
        dist.all_reduce(n)
        tot_valid = int(n.item())
    flops = 2.0 * Tv * V * (d_s + d_t) * 2 + 2.0 * Tv * V * d_s  # forward, recompute, dH
    if args.dw:
        flops += 2.0 * Tv * V * d_s  # dW_s
    peak = 1715.8
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            peak = float(json.load(fh)["bf16_tflops_sustained"])
        peak_kind = "measured (sustained)"
    except Exception:
        peak_kind = "fallback"
    tflops = flops / (call_ms / 1e3) / 1e12
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = fused_cpu_baseline(b, (h_s, W_s, h_t, W_t), step.w[:T])
    out = {"metric": "fused LM-head loss fwd+bwd supervised tokens/s", "value": tot_valid * args.steps / (ms / 1e3),
           "unit": "tokens/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
           "config": {"workload": f"{b.name}_V{V}_ds{d_s}_dt{d_t}", "tokens": T, "supervised_tokens": Tv,
                      "alpha": 1.0, "mode": "full", "flops_per_step": flops,
                      "outputs": "loss, dL/dh_s" + (", dL/dW_s" if args.dw else "")},
           "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak, "unit": "TFLOP/s",
                        "frac": tflops / peak, "peak_kind": peak_kind,
                        "kernel": "turnopd_fused_lmhead_fwd_bwd launch sequence", "launch_ms": call_ms,
                        "traffic": None},
           "gpu_launches": (FUSED_KERNELS_PER_STEP + (1 if args.dw else 0)) * args.steps, "clocks": clocks,
           "e2e": None,
           "cpu_baseline": cpu}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    world, rank, local = dist_env()
    if args.impl == "reference":
        reference_arm(args, world, rank)
        return
    if args.workload == "fused":
        fused_bench(args, world, rank, local)
        return
    import torch

    dist = None
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    import paper_2607_05804_gb300 as P

    P.load()
    b, V, zs, zt, grad, step = build_inputs(args, rank, device)
    R = b.num_valid
    if args.fp32_logits and (args.mode == "topk" or args.vocab_shards):
        raise SystemExit("--fp32-logits times the full-vocabulary and sampled modes")
    if args.vocab_shards:
        if args.mode != "full" or dense_layout(args):
            raise SystemExit("--vocab-shards times the full-vocabulary mode on compact rows")
        step.vp_call = vocab_parallel_loss_fn(step, zs, zt, grad, args.vocab_shards)
    torch.cuda.synchronize()

    for _ in range(max(args.warmup, 3)):
        run_step(step, zs, zt, grad, world, dist)
    torch.cuda.synchronize()
    if step.status() != 0:
        raise RuntimeError(f"device status {step.status()}")

    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(local)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    sampler.start()
    t_start.record()
    for k in range(args.steps):
        run_step(step, zs, zt, grad, world, dist, evs[k])
    t_end.record()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms = t_start.elapsed_time(t_end)
    loss_ms = [a.elapsed_time(z) for a, z in evs]
    if world > 1:
        t = torch.tensor([ms], device=device, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        tot_rows = torch.tensor([R], device=device, dtype=torch.int64)
        dist.all_reduce(tot_rows)
        tot_rows = int(tot_rows.item())
    else:
        tot_rows = R
    if step.status() != 0:
        raise RuntimeError(f"device status {step.status()}")

    value = tot_rows * args.steps / (ms / 1e3)
    peak, peak_kind = load_peaks()
    if args.mode == "topk":
        # teacher row read; the student logits at the K ids; K (id, value) outputs
        bytes_per_row = V * 2 + args.k_top * (2 + 4 + 4)
    elif args.vocab_shards:
        # statistics pass (two logit rows read), gradient pass (read again, gradient written)
        bytes_per_row = 5 * V * 2
    else:
        # two logit rows read (bf16, or fp32) + one gradient row written (bf16, or fp32)
        bytes_per_row = 2 * V * (4 if args.fp32_logits else 2) + V * (4 if args.fp32_grad else 2)
    alg_bytes = R * bytes_per_row
    masked_rows = b.num_tokens - R
    if args.zero_masked:
        # per masked token: a zero gradient row, or (top-K) K ids of -1 and K zero values
        alg_bytes += masked_rows * (args.k_top * (4 + 4) if args.mode == "topk" else V * 2)
    loss_avg_ms = statistics.mean(loss_ms)
    achieved = alg_bytes / (loss_avg_ms / 1e3) / 1e9

    e2e = None
    if not args.no_e2e:
        e2e = e2e_leg(args, step, zs, zt, grad, world, dist, device, R)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(b, zs, zt, V, args.alpha, 0, args.cpu_sample_rows,
                           k_top=args.k_top if args.mode == "topk" else 0, dense=dense_layout(args))

    if rank == 0:
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32" if args.fp32_logits else "bf16",
            "data": "synthetic",
            "config": {
                "workload": f"{b.name}_V{V}", "tokens": b.num_tokens, "supervised_tokens": R,
                "tokens_counted": "supervised (assistant) tokens", "vocab": V,
                "layout": ("dense rows (row i = token i)" if dense_layout(args)
                           else "compact rows (one per supervised token)"),
                **({"zero_masked_grad": True, "masked_rows": masked_rows} if args.zero_masked else {}),
                "grad_dtype": ("fp32 sparse (ids, values)" if args.mode == "topk"
                               else "fp32" if args.fp32_grad else "bf16"),
                "logits_dtype": "fp32" if args.fp32_logits else "bf16",
                "mode": args.mode, "alpha": args.alpha, "scope": "traj",
                **({"k_top": args.k_top} if args.mode == "topk" else {}),
                **({"vocab_shards": args.vocab_shards} if args.vocab_shards else {}),
                "l2": "inputs larger than L2 (%.1f GB streamed per step), no flush" % (alg_bytes / 1e9),
                "packed_tokens_per_s": b.num_tokens * world * args.steps / (ms / 1e3),
            },
            "roofline": {
                "bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "peak_kind": peak_kind,
                "kernel": ("turnopd_topk_loss_fwd_bwd launch sequence (k_topk_rows + compaction + loss sum)"
                           if args.mode == "topk" else
                           f"vocabulary-parallel path, {args.vocab_shards} shards of one GPU "
                           "(shard stats + merge + shard gradients)" if args.vocab_shards else
                           "turnopd_loss_fwd_bwd launch sequence (split-row kernel on clusters of "
                           f"{4 if args.mode == 'sampled' else 8} beside the fp32 helper grid + compaction "
                           "+ loss sum)" if args.fp32_logits else
                           "turnopd_loss_fwd_bwd launch sequence (cluster row kernel beside the helper grid "
                           "+ compaction + loss sum)"),
                "algorithmic_bytes_per_launch": alg_bytes,
                "launch_ms": loss_avg_ms,
                # the committed records cover the full-vocabulary bf16-gradient row grids and the
                # top-K kernel at V = 151,936; any other instantiation or byte count has none
                "traffic": (None if (args.vocab_shards or dense_layout(args) or args.fp32_logits
                                     or V != V_QWEN or args.fp32_grad or args.mode == "sampled")
                            else committed_traffic(args.workload, R, "topk") if args.mode == "topk"
                            else committed_traffic(args.workload)),
            },
            # vocabulary shards: counts(2) + weights(1) + per shard the statistics call (compaction(2),
            # statistics) and the gradient call (compaction(2), gradient, loss sum) + merge + stats(2)
            "gpu_launches": ((KERNELS_PER_STEP + (1 if args.zero_masked else 0)
                              + (0 if args.mode == "topk" else 1))
                             if not args.vocab_shards
                             else 6 + 7 * args.vocab_shards) * args.steps,
            "clocks": clocks,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


def e2e_leg(args, step, zs, zt, grad, world, dist, device, R):
    """Same metric through the public API with inputs in pinned host memory: each
    step copies the logits and batch metadata host->device, runs the step and
    reads the loss back."""
    import torch

    h_zs = torch.empty(zs.shape, dtype=zs.dtype, pin_memory=True)
    h_zt = torch.empty(zt.shape, dtype=zt.dtype, pin_memory=True)
    # Host-resident logits are written by the CPU; pinned pages that only a
    # device->host DMA ever wrote copy back at half the rate on a GB300 host
    # (measured 99 vs 211 GB/s), so the pages are touched from the CPU first.
    h_zs.zero_()
    h_zt.zero_()
    h_zs.copy_(zs)
    h_zt.copy_(zt)
    meta = [step.turn_id, step.loss_mask, step.traj_offsets, step.row_of_token]
    h_meta = [m.cpu().pin_memory() for m in meta]
    h_loss = torch.empty(1, dtype=torch.float64, pin_memory=True)
    steps = max(3, min(args.steps, 10))
    h2d = sum(t.numel() * t.element_size() for t in [h_zs, h_zt] + h_meta)

    # The logits cross in row chunks of about 256 MB, the two models interleaved: on
    # a GB300 host two back-to-back 6 GB cudaMemcpyAsync calls from pinned memory
    # took 115 ms where each alone took 28 ms, and the same bytes in 311 MB chunks
    # took 57 ms (210 GB/s).
    rows_per_chunk = max(1, (256 << 20) // (zs.shape[1] * zs.element_size()))

    def one():
        for r0 in range(0, zs.shape[0], rows_per_chunk):
            r1 = min(zs.shape[0], r0 + rows_per_chunk)
            zs[r0:r1].copy_(h_zs[r0:r1], non_blocking=True)
            zt[r0:r1].copy_(h_zt[r0:r1], non_blocking=True)
        for d, h in zip(meta, h_meta):
            d.copy_(h, non_blocking=True)
        run_step(step, zs, zt, grad, world, dist)
        h_loss.copy_(step.loss, non_blocking=True)

    for _ in range(2):
        one()
    torch.cuda.synchronize()
    a, z = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    a.record()
    for _ in range(steps):
        one()
    z.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(z)
    if world > 1:
        t = torch.tensor([ms], device=device, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return {"value": R * world * steps / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": 8, "steps": steps,
            "d2h": "the loss only: the student-logit gradient stays on the device, where the "
                   "backward pass through the student consumes it"}


if __name__ == "__main__":
    main()
