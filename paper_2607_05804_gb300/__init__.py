"""Python binding of libturnopd, the GB300 (sm_103a) turn-aware OPD loss.

Argument marshalling only: every function forwards torch tensors' device
pointers, sizes and the current CUDA stream to the C entry point of the same
name (``include/turnopd.h``), and raises ``TurnopdError`` on a non-OK status.
All compute runs in the library's CUDA kernels; there is no other path.  If
the library has not been built, importing works but the first call raises.

Build it with ``python -c "import __graft_entry__ as g; g.build()"`` (or
``python paper_2607_05804_gb300/build.py``).
"""
from __future__ import annotations

import ctypes
import os

__all__ = [
    "TurnopdError", "library_path", "load",
    "TURNOPD_FULL_VOCAB", "TURNOPD_SAMPLED_TOKEN", "TURNOPD_F32", "TURNOPD_BF16",
    "TURNOPD_SCOPE_TRAJ", "TURNOPD_SCOPE_BATCH", "TURNOPD_ZERO_MASKED_GRAD",
    "TURNOPD_FORCE_PORTABLE", "TURNOPD_MAX_TURNS",
    "turnopd_turn_counts", "turnopd_weights", "turnopd_weights_workspace_bytes",
    "turnopd_loss_fwd_bwd", "turnopd_loss_workspace_bytes", "turnopd_turn_stats",
    "turnopd_alpha_schedule", "turnopd_turn_floor", "turnopd_status_string", "turnopd_loss_fwd_bwd_static",
    "turnopd_selftest_wait_timeout",
    "TURNOPD_STATIC_MAX_TOKENS", "turnopd_fused_lmhead_fwd_bwd", "turnopd_fused_workspace_bytes",
    "turnopd_topk_loss_fwd_bwd", "TURNOPD_TOPK_MAX", "TURNOPD_TOPK_MAX_VOCAB",
    "turnopd_depth_params", "turnopd_depth_state", "turnopd_depth_default_params",
    "turnopd_depth_init", "turnopd_depth_plan", "turnopd_depth_update", "turnopd_depth_efficiency",
    "turnopd_depth_coverage", "turnopd_turn_diagnostics",
    "turnopd_vocab_stats_bytes", "turnopd_vocab_shard_stats", "turnopd_vocab_stats_merge",
    "turnopd_vocab_shard_loss_grad",
]

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "libturnopd.so")

TURNOPD_FULL_VOCAB, TURNOPD_SAMPLED_TOKEN = 0, 1
TURNOPD_F32, TURNOPD_BF16 = 0, 1
TURNOPD_SCOPE_TRAJ, TURNOPD_SCOPE_BATCH = 0, 1
TURNOPD_ZERO_MASKED_GRAD = 0x1
TURNOPD_FORCE_PORTABLE = 0x100
TURNOPD_MAX_TURNS = 4096
TURNOPD_STATIC_MAX_TOKENS = 65536
TURNOPD_TOPK_MAX = 1024
TURNOPD_TOPK_MAX_VOCAB = 737280

STATUS_NAMES = {
    0: "TURNOPD_OK", 1: "TURNOPD_ERR_NULL", 2: "TURNOPD_ERR_SHAPE", 3: "TURNOPD_ERR_OFFSETS",
    4: "TURNOPD_ERR_TURN_RANGE", 5: "TURNOPD_ERR_TOKEN_RANGE", 6: "TURNOPD_ERR_UNSUPPORTED",
    7: "TURNOPD_ERR_CUDA", 8: "TURNOPD_ERR_TIMEOUT", 9: "TURNOPD_ERR_NONFINITE",
    10: "TURNOPD_ERR_WORKSPACE",
}


class TurnopdError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = int(code)
        super().__init__(f"{where}: {STATUS_NAMES.get(self.code, self.code)} "
                         f"({turnopd_status_string(self.code)})")


def library_path() -> str:
    return _LIB_PATH


_lib = None


def load():
    """Load libturnopd.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(_LIB_PATH):
        raise RuntimeError(f"libturnopd.so not found at {_LIB_PATH}: the CUDA library has not "
                           "been built (run __graft_entry__.build())")
    lib = ctypes.CDLL(_LIB_PATH)
    P, i32, i64, u32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint32
    f64, sz = ctypes.c_double, ctypes.c_size_t
    sig = {
        "turnopd_turn_counts": [P, P, P, i32, i64, i32, P, P, P, P],
        "turnopd_weights": [P, P, P, i32, i64, i32, f64, i32, i32, P, P, P, sz, P, P],
        "turnopd_loss_fwd_bwd": [P, P, i32, i64, i64, i64, P, P, P, P, i64, i32, P, i32, u32,
                                 P, P, P, sz, P, P],
        "turnopd_turn_stats": [P, P, P, P, i32, i64, i32, P, P, P, P, P, P, P],
        "turnopd_loss_fwd_bwd_static": [P, P, i32, i64, i64, i64, P, P, P, P, i64, i32, P, i32,
                                        u32, P, P, P, P],
        "turnopd_fused_lmhead_fwd_bwd": [P, P, i64, P, P, i64, i64, P, P, i64, i32, P, P, P, P, P,
                                         sz, P, P],
        "turnopd_topk_loss_fwd_bwd": [P, P, i32, i64, i64, i64, P, P, P, i64, i32, P, P, P, i32, u32,
                                      P, P, P, sz, P, P],
    }
    D, Pp = ctypes.c_double, ctypes.POINTER
    sig.update({
        "turnopd_depth_default_params": [P],
        "turnopd_depth_init": [P, P],
        "turnopd_depth_plan": [P, P, i64, P, P, P],
        "turnopd_depth_update": [P, P, i64, P, P, P, i32, P, P, i32, P, P],
        "turnopd_depth_efficiency": [P, P, P, i32, D, P, P, P, P],
        "turnopd_depth_coverage": [P, P, i32, D, i32, i32, i32, P],
        "turnopd_turn_diagnostics": [P, P, P, i32, i32, P, P, P],
        "turnopd_vocab_shard_stats": [P, P, i32, i64, i64, i64, P, P, i64, P, P, ctypes.c_size_t, P, P],
        "turnopd_vocab_stats_merge": [P, i32, P, i64, P, P],
        "turnopd_selftest_wait_timeout": [u32, P, P],
        "turnopd_vocab_shard_loss_grad": [P, P, i32, i64, i64, i64, P, P, P, i64, P, P, i32, u32, P, P, P,
                                          sz, P, P],
    })
    for name, args in sig.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    lib.turnopd_weights_workspace_bytes.argtypes = [i32, i32]
    lib.turnopd_weights_workspace_bytes.restype = sz
    lib.turnopd_loss_workspace_bytes.argtypes = [i64]
    lib.turnopd_loss_workspace_bytes.restype = sz
    lib.turnopd_fused_workspace_bytes.argtypes = [i64, i64, i64, i64]
    lib.turnopd_fused_workspace_bytes.restype = sz
    lib.turnopd_alpha_schedule.argtypes = [i64, i64, f64, f64]
    lib.turnopd_alpha_schedule.restype = f64
    lib.turnopd_turn_floor.argtypes = [i64, i32, f64]
    lib.turnopd_turn_floor.restype = i32
    lib.turnopd_depth_default_params.restype = None
    lib.turnopd_vocab_stats_bytes.argtypes = [i64]
    lib.turnopd_vocab_stats_bytes.restype = sz
    lib.turnopd_status_string.argtypes = [ctypes.c_int]
    lib.turnopd_status_string.restype = ctypes.c_char_p
    _lib = lib
    return lib


# ---------------------------------------------------------------- marshalling helpers

def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    import torch

    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, name, dtype=None, numel=None):
    import torch

    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must have dtype {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} needs at least {numel} elements, has {t.numel()}")


def _dtype_code(t, name):
    import torch

    if t.dtype == torch.bfloat16:
        return TURNOPD_BF16
    if t.dtype == torch.float32:
        return TURNOPD_F32
    raise ValueError(f"{name} must be float32 or bfloat16")


def _check(code, where):
    if code != 0:
        raise TurnopdError(code, where)


# ---------------------------------------------------------------- entry points

def turnopd_status_string(code: int) -> str:
    return load().turnopd_status_string(int(code)).decode()


def turnopd_selftest_wait_timeout(poll_limit: int, dev_status, stream=None):
    """One CTA polls a barrier that nothing arrives on; after poll_limit polls it
    records TURNOPD_ERR_TIMEOUT in dev_status (device int32[1])."""
    import torch

    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_selftest_wait_timeout(int(poll_limit), _ptr(dev_status), _stream(stream)),
           "turnopd_selftest_wait_timeout")


def turnopd_alpha_schedule(k: int, K: int, s: float = 0.0, e: float = 1.0) -> float:
    return float(load().turnopd_alpha_schedule(int(k), int(K), float(s), float(e)))


def turnopd_turn_floor(n_traj: int, min_floor: int = 8, min_frac: float = 0.15) -> int:
    """n_min = max(min_floor, ceil(min_frac * n_traj)) for turnopd_weights; defaults
    are the paper's internal-blend settings.  n_traj counts the step's trajectories
    over all ranks."""
    n = int(load().turnopd_turn_floor(int(n_traj), int(min_floor), float(min_frac)))
    if n < 0:
        raise ValueError("turnopd_turn_floor: n_traj and min_floor must be >= 0, min_frac in [0, 1]")
    return n


def turnopd_weights_workspace_bytes(num_traj: int, max_turns: int) -> int:
    return int(load().turnopd_weights_workspace_bytes(int(num_traj), int(max_turns)))


def turnopd_loss_workspace_bytes(num_tokens: int) -> int:
    return int(load().turnopd_loss_workspace_bytes(int(num_tokens)))


def turnopd_fused_workspace_bytes(num_tokens: int, vocab: int, d_s: int, d_t: int) -> int:
    return int(load().turnopd_fused_workspace_bytes(int(num_tokens), int(vocab), int(d_s), int(d_t)))


def turnopd_fused_lmhead_fwd_bwd(h_s, W_s, h_t, W_t, loss_mask, w, mode, dh_s_out, token_loss_out,
                                 loss_out, workspace, dev_status, stream=None, dW_s_out=None):
    """h_s [T, d_s], W_s [V, d_s], h_t [T, d_t], W_t [V, d_t] bf16; dh_s_out [T, d_s] fp32 or
    None; dW_s_out [V, d_s] fp32 or None."""
    import torch

    T, d_s = h_s.shape
    d_t = h_t.shape[1]
    V = W_s.shape[0]
    _need(h_s, "h_s", torch.bfloat16)
    _need(W_s, "W_s", torch.bfloat16)
    _need(h_t, "h_t", torch.bfloat16, T * d_t)
    _need(W_t, "W_t", torch.bfloat16, V * d_t)
    if W_s.shape[1] != d_s or W_t.shape[0] != V or h_t.shape[0] != T:
        raise ValueError("shape mismatch between hidden states and heads")
    _need(loss_mask, "loss_mask", torch.uint8, T)
    _need(w, "w", torch.float32, T)
    _need(dh_s_out, "dh_s_out", torch.float32, T * d_s)
    _need(dW_s_out, "dW_s_out", torch.float32, V * d_s)
    _need(token_loss_out, "token_loss_out", torch.float32, T)
    _need(loss_out, "loss_out", torch.float64, 1)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_fused_lmhead_fwd_bwd(
        _ptr(h_s), _ptr(W_s), d_s, _ptr(h_t), _ptr(W_t), d_t, V, _ptr(loss_mask), _ptr(w), T,
        int(mode), _ptr(dh_s_out), _ptr(dW_s_out), _ptr(token_loss_out), _ptr(loss_out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream)),
        "turnopd_fused_lmhead_fwd_bwd")


def turnopd_turn_counts(turn_id, loss_mask, traj_offsets, max_turns, traj_turn_cnt, counts,
                        dev_status, stream=None):
    import torch

    T, B = turn_id.numel(), traj_offsets.numel() - 1
    _need(turn_id, "turn_id", torch.int32)
    _need(loss_mask, "loss_mask", torch.uint8, T)
    _need(traj_offsets, "traj_offsets", torch.int64)
    _need(traj_turn_cnt, "traj_turn_cnt", torch.int32, B * max_turns)
    _need(counts, "counts", torch.int64, 2 * max_turns + 1)
    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_turn_counts(_ptr(turn_id), _ptr(loss_mask), _ptr(traj_offsets), B, T,
                                      int(max_turns), _ptr(traj_turn_cnt), _ptr(counts),
                                      _ptr(dev_status), _stream(stream)), "turnopd_turn_counts")


def turnopd_weights(turn_id, loss_mask, traj_offsets, max_turns, alpha, scope, n_min,
                    global_counts, w_out, workspace, dev_status, stream=None):
    import torch

    T, B = turn_id.numel(), traj_offsets.numel() - 1
    _need(turn_id, "turn_id", torch.int32)
    _need(loss_mask, "loss_mask", torch.uint8, T)
    _need(traj_offsets, "traj_offsets", torch.int64)
    _need(global_counts, "global_counts", torch.int64, 2 * max_turns + 1)
    _need(w_out, "w_out", torch.float32, T)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_weights(_ptr(turn_id), _ptr(loss_mask), _ptr(traj_offsets), B, T,
                                  int(max_turns), float(alpha), int(scope), int(n_min),
                                  _ptr(global_counts), _ptr(w_out), _ptr(workspace),
                                  workspace.numel() * workspace.element_size(),
                                  _ptr(dev_status), _stream(stream)), "turnopd_weights")


def turnopd_loss_fwd_bwd(z_student, z_teacher, vocab, row_of_token, sampled_ids, loss_mask, w,
                         mode, grad_student, flags, token_loss_out, loss_out, workspace,
                         dev_status, stream=None):
    """z_student, z_teacher: [num_rows, ld] tensors (row stride ld, unit column stride);
    grad_student: None or a tensor of the same shape and strides."""
    import torch

    T = loss_mask.numel()
    for name, z in (("z_student", z_student), ("z_teacher", z_teacher)):
        if not z.is_cuda or z.dim() != 2 or z.stride(1) != 1:
            raise ValueError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if z_teacher.shape != z_student.shape or z_teacher.stride() != z_student.stride() \
            or z_teacher.dtype != z_student.dtype:
        raise ValueError("z_teacher must match z_student in shape, stride and dtype")
    ld = z_student.stride(0)
    if grad_student is not None and (grad_student.shape != z_student.shape
                                     or grad_student.stride(0) != ld or grad_student.stride(1) != 1
                                     or not grad_student.is_cuda):
        raise ValueError("grad_student must match z_student in shape and row stride")
    _need(row_of_token, "row_of_token", torch.int32, T)
    _need(sampled_ids, "sampled_ids", torch.int32, T)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(w, "w", torch.float32, T)
    _need(token_loss_out, "token_loss_out", torch.float32, T)
    _need(loss_out, "loss_out", torch.float64, 1)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    gdt = _dtype_code(grad_student, "grad_student") if grad_student is not None else TURNOPD_F32
    _check(load().turnopd_loss_fwd_bwd(
        _ptr(z_student), _ptr(z_teacher), _dtype_code(z_student, "z_student"), ld, int(vocab),
        z_student.shape[0], _ptr(row_of_token), _ptr(sampled_ids), _ptr(loss_mask), _ptr(w), T,
        int(mode), _ptr(grad_student), gdt, int(flags), _ptr(token_loss_out), _ptr(loss_out),
        _ptr(workspace), workspace.numel() * workspace.element_size(), _ptr(dev_status),
        _stream(stream)), "turnopd_loss_fwd_bwd")


def turnopd_topk_loss_fwd_bwd(z_student, z_teacher, vocab, row_of_token, loss_mask, w, k_top,
                              topk_ids_out, topk_grad_out, grad_student, flags, token_loss_out,
                              loss_out, workspace, dev_status, stream=None):
    """Teacher top-K reverse KL.  z_student, z_teacher: [num_rows, ld] tensors;
    topk_ids_out int32 / topk_grad_out float32 [T, k_top] or None; grad_student None or
    a tensor shaped like z_student."""
    import torch

    T = loss_mask.numel()
    for name, z in (("z_student", z_student), ("z_teacher", z_teacher)):
        if not z.is_cuda or z.dim() != 2 or z.stride(1) != 1:
            raise ValueError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if z_teacher.shape != z_student.shape or z_teacher.stride() != z_student.stride() \
            or z_teacher.dtype != z_student.dtype:
        raise ValueError("z_teacher must match z_student in shape, stride and dtype")
    ld = z_student.stride(0)
    if grad_student is not None and (grad_student.shape != z_student.shape
                                     or grad_student.stride(0) != ld or grad_student.stride(1) != 1
                                     or not grad_student.is_cuda):
        raise ValueError("grad_student must match z_student in shape and row stride")
    _need(row_of_token, "row_of_token", torch.int32, T)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(w, "w", torch.float32, T)
    _need(topk_ids_out, "topk_ids_out", torch.int32, T * int(k_top))
    _need(topk_grad_out, "topk_grad_out", torch.float32, T * int(k_top))
    _need(token_loss_out, "token_loss_out", torch.float32, T)
    _need(loss_out, "loss_out", torch.float64, 1)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    gdt = _dtype_code(grad_student, "grad_student") if grad_student is not None else TURNOPD_F32
    _check(load().turnopd_topk_loss_fwd_bwd(
        _ptr(z_student), _ptr(z_teacher), _dtype_code(z_student, "z_student"), ld, int(vocab),
        z_student.shape[0], _ptr(row_of_token), _ptr(loss_mask), _ptr(w), T, int(k_top),
        _ptr(topk_ids_out), _ptr(topk_grad_out), _ptr(grad_student), gdt, int(flags),
        _ptr(token_loss_out), _ptr(loss_out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream)),
        "turnopd_topk_loss_fwd_bwd")


# ---------------------------------------------------------------- vocabulary-parallel split

def _shard_logits(z_student, z_teacher):
    for name, z in (("z_student", z_student), ("z_teacher", z_teacher)):
        if not z.is_cuda or z.dim() != 2 or z.stride(1) != 1:
            raise ValueError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if z_teacher.shape != z_student.shape or z_teacher.stride() != z_student.stride() \
            or z_teacher.dtype != z_student.dtype:
        raise ValueError("z_teacher must match z_student in shape, stride and dtype")
    return z_student.stride(0), z_student.shape[1]


def turnopd_vocab_stats_bytes(num_tokens: int) -> int:
    return int(load().turnopd_vocab_stats_bytes(int(num_tokens)))


def turnopd_vocab_shard_stats(z_student, z_teacher, row_of_token, loss_mask, stats_out, workspace, dev_status,
                              stream=None):
    """z_student, z_teacher: this rank's [num_rows, shard_vocab] column shard (row stride ld);
    stats_out float32 [T, 6]; workspace of turnopd_loss_workspace_bytes(T) bytes."""
    import torch

    ld, Vr = _shard_logits(z_student, z_teacher)
    T = loss_mask.numel()
    _need(row_of_token, "row_of_token", torch.int32, T)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(stats_out, "stats_out", torch.float32, T * 6)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_vocab_shard_stats(
        _ptr(z_student), _ptr(z_teacher), _dtype_code(z_student, "z_student"), ld, Vr, z_student.shape[0],
        _ptr(row_of_token), _ptr(loss_mask), T, _ptr(stats_out), _ptr(workspace),
        workspace.numel() * workspace.element_size(), _ptr(dev_status), _stream(stream)),
        "turnopd_vocab_shard_stats")


def turnopd_vocab_stats_merge(parts, loss_mask, merged_out, stream=None):
    """parts float32 [n_shards, T, 6] (shard order) -> merged_out [T, 6]."""
    import torch

    T = loss_mask.numel()
    _need(parts, "parts", torch.float32)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(merged_out, "merged_out", torch.float32, T * 6)
    _check(load().turnopd_vocab_stats_merge(_ptr(parts), parts.shape[0], _ptr(loss_mask), T, _ptr(merged_out),
                                            _stream(stream)), "turnopd_vocab_stats_merge")


def turnopd_vocab_shard_loss_grad(z_student, z_teacher, row_of_token, loss_mask, w, merged_stats, grad_shard,
                                  flags, token_loss_out, loss_out, workspace, dev_status, stream=None):
    import torch

    ld, Vr = _shard_logits(z_student, z_teacher)
    T = loss_mask.numel()
    if grad_shard is not None and (grad_shard.shape != z_student.shape or grad_shard.stride(0) != ld
                                   or grad_shard.stride(1) != 1 or not grad_shard.is_cuda):
        raise ValueError("grad_shard must match the logit shard in shape and row stride")
    _need(row_of_token, "row_of_token", torch.int32, T)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(w, "w", torch.float32, T)
    _need(merged_stats, "merged_stats", torch.float32, T * 6)
    _need(token_loss_out, "token_loss_out", torch.float32, T)
    _need(loss_out, "loss_out", torch.float64, 1)
    _need(workspace, "workspace")
    _need(dev_status, "dev_status", torch.int32, 1)
    gdt = _dtype_code(grad_shard, "grad_shard") if grad_shard is not None else TURNOPD_F32
    _check(load().turnopd_vocab_shard_loss_grad(
        _ptr(z_student), _ptr(z_teacher), _dtype_code(z_student, "z_student"), ld, Vr, z_student.shape[0],
        _ptr(row_of_token), _ptr(loss_mask), _ptr(w), T, _ptr(merged_stats), _ptr(grad_shard), gdt, int(flags),
        _ptr(token_loss_out), _ptr(loss_out), _ptr(workspace), workspace.numel() * workspace.element_size(),
        _ptr(dev_status), _stream(stream)), "turnopd_vocab_shard_loss_grad")


# ---------------------------------------------------------------- rollout-depth controller (host)

class turnopd_depth_params(ctypes.Structure):
    _fields_ = [("h_min", ctypes.c_int32), ("h_max", ctypes.c_int32), ("ema_alpha", ctypes.c_double),
                ("coverage_p", ctypes.c_double), ("min_cov_traj", ctypes.c_int32),
                ("use_success", ctypes.c_int32), ("warmup_steps", ctypes.c_int32),
                ("probe_interval", ctypes.c_int32), ("eps", ctypes.c_double)]


class turnopd_depth_state(ctypes.Structure):
    _fields_ = [("h_bar", ctypes.c_double), ("h_eff_bar", ctypes.c_double), ("h_eff", ctypes.c_int32),
                ("h_cov", ctypes.c_int32), ("h_ctrl", ctypes.c_int32)]


def _host(a, dtype):
    import numpy as np

    if hasattr(a, "detach"):  # torch tensor (any device): copied to host memory
        a = a.detach().cpu().numpy()
    return np.ascontiguousarray(a, dtype=dtype)


def _hp(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def turnopd_depth_default_params() -> turnopd_depth_params:
    p = turnopd_depth_params()
    load().turnopd_depth_default_params(ctypes.byref(p))
    return p


def turnopd_depth_init(params: turnopd_depth_params) -> turnopd_depth_state:
    st = turnopd_depth_state()
    _check(load().turnopd_depth_init(ctypes.byref(params), ctypes.byref(st)), "turnopd_depth_init")
    return st


def turnopd_depth_plan(params, state, k: int):
    """-> (h_hat, is_probe, h_roll) for step k (1-based)."""
    h, pr, roll = ctypes.c_int32(), ctypes.c_int32(), ctypes.c_int32()
    _check(load().turnopd_depth_plan(ctypes.byref(params), ctypes.byref(state), int(k), ctypes.byref(h),
                                     ctypes.byref(pr), ctypes.byref(roll)), "turnopd_depth_plan")
    return h.value, bool(pr.value), roll.value


def turnopd_depth_update(params, state, k: int, turn_sum, turn_cnt, turn_surv, traj_len, traj_success,
                         want_mq=False):
    """Host arrays (numpy or torch, copied to host).  Updates `state` in place; returns
    (m, q) when want_mq."""
    import numpy as np

    ts, tc, sv = _host(turn_sum, np.float64), _host(turn_cnt, np.int64), _host(turn_surv, np.int32)
    tl, su = _host(traj_len, np.int32), _host(traj_success, np.uint8)
    T = ts.size
    m = np.zeros(max(T, 1)) if want_mq else None
    q = np.zeros(max(T, 1)) if want_mq else None
    _check(load().turnopd_depth_update(ctypes.byref(params), ctypes.byref(state), int(k), _hp(ts), _hp(tc),
                                       _hp(sv), T, _hp(tl), _hp(su), tl.size, _hp(m), _hp(q)),
           "turnopd_depth_update")
    return (m[:T], q[:T]) if want_mq else None


def turnopd_depth_efficiency(turn_sum, turn_cnt, turn_surv, eps=1e-8):
    """-> (m, q, h_eff_bar, h_eff)."""
    import numpy as np

    ts, tc, sv = _host(turn_sum, np.float64), _host(turn_cnt, np.int64), _host(turn_surv, np.int32)
    T = ts.size
    m, q = np.zeros(max(T, 1)), np.zeros(max(T, 1))
    hb, he = ctypes.c_double(), ctypes.c_int32()
    _check(load().turnopd_depth_efficiency(_hp(ts), _hp(tc), _hp(sv), T, float(eps), _hp(m), _hp(q),
                                           ctypes.byref(hb), ctypes.byref(he)), "turnopd_depth_efficiency")
    return m[:T], q[:T], hb.value, he.value


def turnopd_depth_coverage(traj_len, traj_success, p=0.8, min_cov_traj=8, use_success=True, previous=0):
    import numpy as np

    tl, su = _host(traj_len, np.int32), _host(traj_success, np.uint8)
    h = ctypes.c_int32()
    _check(load().turnopd_depth_coverage(_hp(tl), _hp(su), tl.size, float(p), int(min_cov_traj),
                                         int(bool(use_success)), int(previous), ctypes.byref(h)),
           "turnopd_depth_coverage")
    return h.value


def turnopd_turn_diagnostics(turn_sum, turn_cnt, turn_surv, n_min=1):
    """-> (b [T], s [T], deep [4] = prefix, deep/shallow KL ratio, deep support, deep loss budget)."""
    import numpy as np

    ts, tc, sv = _host(turn_sum, np.float64), _host(turn_cnt, np.int64), _host(turn_surv, np.int32)
    T = ts.size
    b, sh, deep = np.zeros(max(T, 1)), np.zeros(max(T, 1)), np.zeros(4)
    _check(load().turnopd_turn_diagnostics(_hp(ts), _hp(tc), _hp(sv), T, int(n_min), _hp(b), _hp(sh),
                                           _hp(deep)), "turnopd_turn_diagnostics")
    return b[:T], sh[:T], deep


def turnopd_turn_stats(token_loss, turn_id, loss_mask, traj_offsets, max_turns, traj_turn_sum,
                       traj_turn_cnt, turn_sum, turn_cnt, turn_surv, dev_status, stream=None):
    import torch

    T, B = turn_id.numel(), traj_offsets.numel() - 1
    _need(token_loss, "token_loss", torch.float32, T)
    _need(turn_id, "turn_id", torch.int32)
    _need(loss_mask, "loss_mask", torch.uint8, T)
    _need(traj_offsets, "traj_offsets", torch.int64)
    _need(traj_turn_sum, "traj_turn_sum", torch.float64, B * max_turns)
    _need(traj_turn_cnt, "traj_turn_cnt", torch.int32, B * max_turns)
    _need(turn_sum, "turn_sum", torch.float64, max_turns)
    _need(turn_cnt, "turn_cnt", torch.int64, max_turns)
    _need(turn_surv, "turn_surv", torch.int32, max_turns)
    _need(dev_status, "dev_status", torch.int32, 1)
    _check(load().turnopd_turn_stats(_ptr(token_loss), _ptr(turn_id), _ptr(loss_mask),
                                     _ptr(traj_offsets), B, T, int(max_turns), _ptr(traj_turn_sum),
                                     _ptr(traj_turn_cnt), _ptr(turn_sum), _ptr(turn_cnt),
                                     _ptr(turn_surv), _ptr(dev_status), _stream(stream)),
           "turnopd_turn_stats")


def turnopd_loss_fwd_bwd_static(z_student, z_teacher, vocab, row_of_token, sampled_ids, loss_mask,
                                w, mode, grad_student, flags, token_loss_out, loss_out, dev_status,
                                stream=None):
    """turnopd_loss_fwd_bwd without a workspace argument, for callers that cannot
    allocate device memory: the library's own static device scratch is used instead
    (at most TURNOPD_STATIC_MAX_TOKENS tokens; calls must not overlap on the GPU)."""
    import torch

    T = loss_mask.numel()
    for name, z in (("z_student", z_student), ("z_teacher", z_teacher)):
        if not z.is_cuda or z.dim() != 2 or z.stride(1) != 1:
            raise ValueError(f"{name} must be a 2-D CUDA tensor with unit column stride")
    if z_teacher.shape != z_student.shape or z_teacher.stride() != z_student.stride() \
            or z_teacher.dtype != z_student.dtype:
        raise ValueError("z_teacher must match z_student in shape, stride and dtype")
    ld = z_student.stride(0)
    if grad_student is not None and (grad_student.shape != z_student.shape
                                     or grad_student.stride(0) != ld or grad_student.stride(1) != 1
                                     or not grad_student.is_cuda):
        raise ValueError("grad_student must match z_student in shape and row stride")
    _need(row_of_token, "row_of_token", torch.int32, T)
    _need(sampled_ids, "sampled_ids", torch.int32, T)
    _need(loss_mask, "loss_mask", torch.uint8)
    _need(w, "w", torch.float32, T)
    _need(token_loss_out, "token_loss_out", torch.float32, T)
    _need(loss_out, "loss_out", torch.float64, 1)
    _need(dev_status, "dev_status", torch.int32, 1)
    gdt = _dtype_code(grad_student, "grad_student") if grad_student is not None else TURNOPD_F32
    _check(load().turnopd_loss_fwd_bwd_static(
        _ptr(z_student), _ptr(z_teacher), _dtype_code(z_student, "z_student"), ld, int(vocab),
        z_student.shape[0], _ptr(row_of_token), _ptr(sampled_ids), _ptr(loss_mask), _ptr(w), T,
        int(mode), _ptr(grad_student), gdt, int(flags), _ptr(token_loss_out), _ptr(loss_out),
        _ptr(dev_status), _stream(stream)), "turnopd_loss_fwd_bwd_static")
