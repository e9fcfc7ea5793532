"""Seeded synthetic inputs for the turn-aware OPD loss.

This module only draws random numbers and lays out packed batches: it holds
none of the loss arithmetic, and both the CUDA path and the CPU oracle take
their inputs from it.  The paper's agent workloads (ALFWorld household tasks,
Multi-Hop Search, WebShop) are stood in for by the five shapes below; no item
of those datasets is reproduced.

Packed-batch layout: trajectory b owns tokens [traj_offsets[b],
traj_offsets[b+1]); inside it spans alternate [obs_0, asst_0, obs_1, asst_1,
...].  Observation tokens have loss_mask = 0 and turn_id = -1; the tokens of
the k-th assistant span have loss_mask = 1 and turn_id = k (0-based turns).

Logit rows are either dense (row i belongs to token i) or compact (one row per
supervised token, in token order; row_of_token[i] = -1 for masked tokens).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

V_QWEN = 151_936


@dataclass
class Batch:
    name: str
    turn_id: np.ndarray        # int32 [T]
    loss_mask: np.ndarray      # uint8 [T]
    traj_offsets: np.ndarray   # int64 [B+1]
    max_turns: int
    info: dict = field(default_factory=dict)

    @property
    def num_tokens(self) -> int:
        return int(self.turn_id.size)

    @property
    def num_traj(self) -> int:
        return int(self.traj_offsets.size - 1)

    @property
    def num_valid(self) -> int:
        return int(self.loss_mask.sum())

    def compact_rows(self) -> np.ndarray:
        """row_of_token for the compact layout (rows only for supervised tokens)."""
        rot = np.full(self.num_tokens, -1, np.int32)
        idx = np.nonzero(self.loss_mask)[0]
        rot[idx] = np.arange(idx.size, dtype=np.int32)
        return rot


def _from_spans(name, traj_spans, max_turns, info=None) -> Batch:
    """traj_spans: list (per trajectory) of lists of (kind, length), kind 'o'/'a'/'p'."""
    tid, msk, off = [], [], [0]
    for spans in traj_spans:
        turn = 0
        n = 0
        for kind, length in spans:
            if length <= 0:
                continue
            if kind == "a":
                tid.append(np.full(length, turn, np.int32))
                msk.append(np.ones(length, np.uint8))
                turn += 1
            else:
                tid.append(np.full(length, -1, np.int32))
                msk.append(np.zeros(length, np.uint8))
            n += length
        off.append(off[-1] + n)
    turn_id = np.concatenate(tid) if tid else np.zeros(0, np.int32)
    loss_mask = np.concatenate(msk) if msk else np.zeros(0, np.uint8)
    return Batch(name, turn_id, loss_mask, np.asarray(off, np.int64), max_turns, info or {})


def _fit_total(lengths, total):
    """Rescale integer span lengths proportionally so they sum to exactly `total`."""
    lengths = np.asarray(lengths, np.int64)
    cum = np.cumsum(lengths)
    new_cum = np.round(cum * (total / cum[-1])).astype(np.int64)
    new_cum[-1] = total
    return np.diff(np.concatenate([[0], new_cum]))


def tiny(seed: int = 0) -> Batch:
    """2 trajectories x 4 turns of [16 observation, 16 assistant] tokens (T = 256)."""
    spans = [[("o", 16), ("a", 16)] * 4 for _ in range(2)]
    return _from_spans("tiny_2x128", spans, max_turns=4)


def packed(seed: int = 0, num_traj: int = 8, traj_len: int = 4096) -> Batch:
    """8 x 4096 tokens; 10-30 turns; turn length ~ Geometric(1/150) split 40 % observation,
    spans rescaled to fill each trajectory exactly."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(num_traj):
        n_turns = int(rng.integers(10, 31))
        L = rng.geometric(1.0 / 150.0, size=n_turns)
        obs = np.round(0.4 * L).astype(np.int64)
        asst = np.maximum(L - obs, 1)
        inter = np.empty(2 * n_turns, np.int64)
        inter[0::2], inter[1::2] = obs, asst
        fit = _fit_total(inter, traj_len)
        # every assistant span keeps at least one token
        for k in range(1, fit.size, 2):
            if fit[k] < 1:
                j = int(np.argmax(fit[0::2])) * 2
                fit[j] -= 1
                fit[k] += 1
        out.append([("o" if k % 2 == 0 else "a", int(x)) for k, x in enumerate(fit)])
    return _from_spans(f"packed_{num_traj}x{traj_len}", out, max_turns=30)


def household(seed: int = 0, num_traj: int = 16, traj_len: int = 8192) -> Batch:
    """16 x 8192 tokens; up to 50 turns; observations U[100,300], actions U[10,40];
    truncated at the trajectory length, masked padding after the last turn."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(num_traj):
        n_turns = int(rng.integers(10, 51))
        spans, total = [], 0
        for _t in range(n_turns):
            for kind, length in (("o", int(rng.integers(100, 301))), ("a", int(rng.integers(10, 41)))):
                if total >= traj_len:
                    break
                length = min(length, traj_len - total)
                spans.append((kind, length))
                total += length
        if total < traj_len:
            spans.append(("p", traj_len - total))
        out.append(spans)
    return _from_spans(f"household_{num_traj}x{traj_len}", out, max_turns=50)


def multihop(seed: int = 0, num_traj: int = 64, min_len: int = 512, max_len: int = 16384) -> Batch:
    """64 ragged trajectories, lengths U[512, 16384]; 2-12 turns; observations U[200,1500];
    assistant spans min(floor(8 (1 + Pareto(1.5))), 2000) (heavy tailed)."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(num_traj):
        L = int(rng.integers(min_len, max_len + 1))
        n_turns = int(rng.integers(2, 13))
        obs = rng.integers(200, 1501, size=n_turns).astype(np.int64)
        asst = np.minimum(np.floor(8.0 * (1.0 + rng.pareto(1.5, size=n_turns))), 2000).astype(np.int64)
        total = int(obs.sum() + asst.sum())
        if total < L:
            obs = _fit_total(obs, L - int(asst.sum()))
        spans, acc = [], 0
        for o, a in zip(obs, asst):
            for kind, length in (("o", int(o)), ("a", int(a))):
                if acc >= L:
                    break
                length = min(length, L - acc)
                spans.append((kind, length))
                acc += length
        out.append(spans)
    return _from_spans(f"multihop_{num_traj}", out, max_turns=12)


def fused(seed: int = 0, num_traj: int = 8, traj_len: int = 2048) -> Batch:
    """Fused LM-head case: 8 x 2048 tokens with the packed-batch turn structure."""
    b = packed(seed, num_traj=num_traj, traj_len=traj_len)
    b.name = f"fused_{num_traj}x{traj_len}"
    return b


def random_structure(rng: np.random.Generator, num_traj: int, max_len: int, max_turns: int,
                     p_mask: float = 0.4, allow_empty: bool = True) -> Batch:
    """Small random packed batch for property tests: runs of masked/unmasked tokens,
    turn ids increasing by run, some trajectories possibly empty or fully masked."""
    spans_all = []
    for _ in range(num_traj):
        L = int(rng.integers(0 if allow_empty else 1, max_len + 1))
        spans, acc, turns = [], 0, 0
        while acc < L:
            length = int(min(rng.integers(1, 9), L - acc))
            kind = "o" if (rng.random() < p_mask or turns >= max_turns) else "a"
            if kind == "a":
                turns += 1
            spans.append((kind, length))
            acc += length
        spans_all.append(spans)
    return _from_spans("random", spans_all, max_turns=max_turns)


CONFIGS = {
    "tiny": tiny,
    "packed": packed,
    "household": household,
    "multihop": multihop,
    "fused": fused,
}


# ---------------------------------------------------------------- logits

def make_logits(num_rows: int, vocab: int, kind: str, dtype, seed: int, device="cpu",
                ld: int | None = None, chunk_rows: int = 1024):
    """Student and teacher logits [num_rows, ld] (first `vocab` columns used).

    kind "tiny":  z_s ~ N(0, 2^2), z_t = z_s + N(0, 0.5^2).
    kind "agent": base ~ N(0, 3^2); z_s = base, z_t = 0.8 base + 0.6 N(0, 3^2)
                  (correlation 0.8, equal variance); 5 distinct ids per row get +8
                  in both models (a shared peaked component).
    Drawn in fp32 with a torch generator on `device`, then cast to `dtype`.
    """
    import torch

    ld = vocab if ld is None else ld
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    zs = torch.empty((num_rows, ld), dtype=dtype, device=device)
    zt = torch.empty((num_rows, ld), dtype=dtype, device=device)
    if ld > vocab:
        zs[:, vocab:] = 0
        zt[:, vocab:] = 0
    for r0 in range(0, num_rows, chunk_rows):
        r1 = min(num_rows, r0 + chunk_rows)
        n = r1 - r0
        if kind == "tiny":
            a = torch.randn((n, vocab), generator=gen, device=device) * 2.0
            b = a + torch.randn((n, vocab), generator=gen, device=device) * 0.5
        elif kind == "agent":
            base = torch.randn((n, vocab), generator=gen, device=device) * 3.0
            noise = torch.randn((n, vocab), generator=gen, device=device) * 3.0
            a = base
            b = 0.8 * base + 0.6 * noise
            ids = torch.multinomial(torch.ones((n, vocab), device=device), 5,
                                    replacement=False, generator=gen)
            a.scatter_add_(1, ids, torch.full(ids.shape, 8.0, device=device))
            b.scatter_add_(1, ids, torch.full(ids.shape, 8.0, device=device))
        else:
            raise ValueError(kind)
        zs[r0:r1, :vocab] = a.to(dtype)
        zt[r0:r1, :vocab] = b.to(dtype)
    return zs, zt


def sample_ids(z_student, seed: int, vocab: int | None = None, chunk_rows: int = 1024):
    """y ~ softmax(z_student) per row by the Gumbel-max rule (exact sampling)."""
    import torch

    vocab = z_student.shape[1] if vocab is None else vocab
    gen = torch.Generator(device=z_student.device)
    gen.manual_seed(seed)
    out = torch.empty(z_student.shape[0], dtype=torch.int32, device=z_student.device)
    for r0 in range(0, z_student.shape[0], chunk_rows):
        r1 = min(z_student.shape[0], r0 + chunk_rows)
        z = z_student[r0:r1, :vocab].float()
        u = torch.rand(z.shape, generator=gen, device=z.device).clamp_(1e-20, 1.0)
        out[r0:r1] = torch.argmax(z - torch.log(-torch.log(u)), dim=1).to(torch.int32)
    return out


def make_fused(num_tokens: int, d_s: int, d_t: int, vocab: int, seed: int, device="cpu"):
    """h_s ~ N(0,1) [T, d_s], W_s ~ N(0, 0.02^2) [V, d_s], and likewise for the teacher,
    all bf16."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    bf = torch.bfloat16

    def draw(shape, std):
        out = torch.empty(shape, dtype=bf, device=device)
        rows = max(1, (1 << 26) // shape[1])
        for r0 in range(0, shape[0], rows):
            r1 = min(shape[0], r0 + rows)
            out[r0:r1] = (torch.randn((r1 - r0, shape[1]), generator=gen, device=device) * std).to(bf)
        return out

    h_s = draw((num_tokens, d_s), 1.0)
    W_s = draw((vocab, d_s), 0.02)
    h_t = draw((num_tokens, d_t), 1.0)
    W_t = draw((vocab, d_t), 0.02)
    return h_s, W_s, h_t, W_t


def bf16_bits(t):
    """numpy uint16 view of a bf16 torch tensor's bits (CPU copy)."""
    import torch

    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
