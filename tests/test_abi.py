"""The C-ABI library loads and exports every symbol include/turnopd.h declares,
and its host-side argument checks answer without a GPU (they return before any
CUDA call).  No compute call is made here."""
import ctypes
import math
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "turnopd.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_05804_gb300 import build as B

    B.build()
    import paper_2607_05804_gb300 as P

    return P.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^[A-Za-z_][\w \*]*?\b(turnopd_\w+)\s*\(", src, flags=re.M)))


def test_header_declares_the_entry_points():
    names = declared_functions()
    for n in ("turnopd_turn_counts", "turnopd_weights", "turnopd_loss_fwd_bwd",
              "turnopd_turn_stats", "turnopd_alpha_schedule", "turnopd_status_string",
              "turnopd_weights_workspace_bytes", "turnopd_loss_workspace_bytes"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_binding_names_match_header():
    import paper_2607_05804_gb300 as P

    for n in declared_functions():
        assert hasattr(P, n), n


FAKE = ctypes.c_void_p(0x10000)  # never dereferenced: every call below fails validation first


def test_loss_host_validation(lib):
    P = ctypes.c_void_p
    f = lib.turnopd_loss_fwd_bwd
    ws_need = lib.turnopd_loss_workspace_bytes(64)
    assert ws_need > 0

    def call(zs=FAKE, ld=1024, vocab=1024, rows=64, T=64, mode=0, grad_dtype=0, in_dtype=1,
             flags=0, ws=FAKE, wsb=None, loss=FAKE, status=FAKE, y=FAKE, grad=FAKE):
        return f(zs, FAKE, in_dtype, ld, vocab, rows, None, y, FAKE, FAKE, T, mode, grad,
                 grad_dtype, flags, FAKE, loss, ws, ws_need if wsb is None else wsb, status, None)

    assert call(zs=None) == 1
    assert call(loss=None) == 1
    assert call(status=None) == 1
    assert call(mode=1, y=None) == 1
    assert call(ld=100, vocab=101) == 2
    assert call(vocab=0) == 2
    assert call(rows=10) == 2          # dense rows need num_rows >= num_tokens
    assert call(mode=7) == 6
    assert call(in_dtype=5) == 6
    assert call(grad_dtype=3) == 6
    assert call(flags=0x8000) == 6
    assert call(ws=None) == 10
    assert call(wsb=ws_need - 1) == 10
    assert call(ws=ctypes.c_void_p(0x10010)) == 10  # not 256-byte aligned
    assert call(zs=ctypes.c_void_p(0x10001)) == 2   # misaligned bf16 pointer


def test_structure_host_validation(lib):
    f = lib.turnopd_weights
    need = lib.turnopd_weights_workspace_bytes(4, 8)
    base = dict(tid=FAKE, msk=FAKE, off=FAKE, B=4, T=100, Tm=8, alpha=0.5, scope=0, n_min=0,
                w=FAKE, ws=FAKE, wsb=need, st=FAKE)

    def call(**kw):
        a = dict(base, **kw)
        return f(a["tid"], a["msk"], a["off"], a["B"], a["T"], a["Tm"], a["alpha"], a["scope"],
                 a["n_min"], None, a["w"], a["ws"], a["wsb"], a["st"], None)

    assert call(off=None) == 1
    assert call(st=None) == 1
    assert call(w=None) == 1
    assert call(Tm=0) == 2
    assert call(Tm=5000) == 2
    assert call(B=-1) == 2
    assert call(alpha=1.5) == 2
    assert call(alpha=float("nan")) == 2
    assert call(scope=9) == 6
    assert call(wsb=need - 1) == 10
    g = lib.turnopd_turn_stats
    assert g(None, FAKE, FAKE, FAKE, 4, 100, 8, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None) == 1
    assert g(FAKE, FAKE, FAKE, FAKE, 4, 100, 8, FAKE, FAKE, None, FAKE, FAKE, FAKE, None) == 1
    h = lib.turnopd_turn_counts
    assert h(FAKE, FAKE, FAKE, 4, 100, 8, FAKE, None, FAKE, None) == 1


def test_alpha_schedule_and_status_strings(lib, oracle):
    import paper_2607_05804_gb300 as P

    for k in range(0, 101, 7):
        assert P.turnopd_alpha_schedule(k, 100) == oracle.alpha_schedule(k, 100)
    assert math.isnan(P.turnopd_alpha_schedule(1, 0))
    assert math.isnan(P.turnopd_alpha_schedule(1, 10, 0.5, 0.5))
    for code in range(11):
        assert P.turnopd_status_string(code)
    assert P.turnopd_status_string(0) == "ok"


def test_turn_floor_is_the_paper_rule_with_an_exact_ceiling(lib):
    """n_min = max(floor, ceil(frac * n_traj)) (hyper-parameter table: floor 8,
    frac 0.15), checked against exact rational arithmetic on the decimal frac."""
    from fractions import Fraction

    import paper_2607_05804_gb300 as P

    for frac in ("0.15", "0.1", "0.3", "0.25", "0.07", "1", "0"):
        for floor in (0, 8):
            for n in list(range(0, 201)) + [1000, 4096, 65536, 10 ** 7]:
                want = max(floor, math.ceil(Fraction(frac) * n))
                assert P.turnopd_turn_floor(n, floor, float(frac)) == want, (frac, floor, n)
    assert P.turnopd_turn_floor(64) == 10          # the paper's batch of 64 trajectories
    assert P.turnopd_turn_floor(16) == 8           # household: the floor binds
    assert 0.07 * 100 > 7 and P.turnopd_turn_floor(100, 0, 0.07) == 7
    for bad in ((-1, 8, 0.15), (10, -1, 0.15), (10, 8, -0.1), (10, 8, 1.5), (10, 8, float("nan"))):
        assert lib.turnopd_turn_floor(*bad) == -1
    with pytest.raises(ValueError):
        P.turnopd_turn_floor(-1)


def test_topk_host_validation(lib):
    f = lib.turnopd_topk_loss_fwd_bwd
    ws_need = lib.turnopd_loss_workspace_bytes(64)

    def call(zs=FAKE, ld=1024, vocab=1024, rows=64, T=64, k=50, in_dtype=1, grad_dtype=0,
             flags=0, ws=FAKE, wsb=None, loss=FAKE, status=FAKE, ids=FAKE, g=FAKE, grad=None):
        return f(zs, FAKE, in_dtype, ld, vocab, rows, None, FAKE, FAKE, T, k, ids, g, grad,
                 grad_dtype, flags, FAKE, loss, ws, ws_need if wsb is None else wsb, status, None)

    assert call(zs=None) == 1
    assert call(loss=None) == 1
    assert call(status=None) == 1
    assert call(k=0) == 2
    assert call(k=1025) == 2
    assert call(k=51, vocab=50, ld=64) == 2          # k_top > vocab
    assert call(vocab=737280 + 1, ld=737280 + 8) == 2
    assert call(ld=100, vocab=101) == 2
    assert call(rows=10) == 2
    assert call(ids=ctypes.c_void_p(0x10002)) == 2   # misaligned int32 output
    assert call(in_dtype=5) == 6
    assert call(grad=FAKE, grad_dtype=4) == 6
    assert call(flags=0x100) == 6                     # only TURNOPD_ZERO_MASKED_GRAD
    assert call(ws=None) == 10
    assert call(wsb=ws_need - 1) == 10


def test_vocab_shard_host_validation(lib):
    f = lib.turnopd_vocab_shard_stats
    ws_need = lib.turnopd_loss_workspace_bytes(64)

    def call(zs=FAKE, ld=1024, vocab=1024, rows=64, T=64, in_dtype=1, stats=FAKE, ws=FAKE, wsb=None,
             status=FAKE):
        return f(zs, FAKE, in_dtype, ld, vocab, rows, None, FAKE, T, stats, ws,
                 ws_need if wsb is None else wsb, status, None)

    assert call(zs=None) == 1
    assert call(status=None) == 1
    assert call(stats=None) == 1
    assert call(in_dtype=5) == 6
    assert call(ld=100, vocab=101) == 2
    assert call(rows=63) == 2                        # no row map: a row per token
    assert call(stats=ctypes.c_void_p(0x10002)) == 2  # misaligned float32 output
    assert call(ws=None) == 10
    assert call(wsb=ws_need - 1) == 10
    assert call(ws=ctypes.c_void_p(0x10010)) == 10    # not 256-byte aligned


def test_vocab_merge_and_shard_grad_host_validation(lib):
    merge = lib.turnopd_vocab_stats_merge
    assert merge(None, 2, FAKE, 64, FAKE, None) == 1
    assert merge(FAKE, 2, FAKE, 64, None, None) == 1
    assert merge(FAKE, 0, FAKE, 64, FAKE, None) == 2                    # no shard
    assert merge(FAKE, 2, FAKE, -1, FAKE, None) == 2
    assert merge(ctypes.c_void_p(0x10002), 2, FAKE, 64, FAKE, None) == 2  # misaligned float32 partials
    assert merge(None, 2, None, 0, None, None) == 0                     # nothing to merge, no launch

    f = lib.turnopd_vocab_shard_loss_grad
    ws_need = lib.turnopd_loss_workspace_bytes(64)

    def call(zs=FAKE, ld=1024, vocab=1024, rows=64, T=64, in_dtype=1, stats=FAKE, grad=FAKE, grad_dtype=1,
             flags=0, tl=FAKE, loss=FAKE, ws=FAKE, wsb=None, status=FAKE):
        return f(zs, FAKE, in_dtype, ld, vocab, rows, None, FAKE, FAKE, T, stats, grad, grad_dtype, flags, tl,
                 loss, ws, ws_need if wsb is None else wsb, status, None)

    assert call(zs=None) == 1
    assert call(status=None) == 1
    assert call(loss=None) == 1
    assert call(stats=None) == 1
    assert call(tl=None) == 1
    assert call(in_dtype=3) == 6
    assert call(grad_dtype=2) == 6
    assert call(flags=0x2) == 6
    assert call(ld=512) == 2                                            # ld < shard width
    assert call(grad=ctypes.c_void_p(0x10001)) == 2                     # misaligned bf16 gradient
    assert call(loss=ctypes.c_void_p(0x10004)) == 2                     # misaligned fp64 loss
    assert call(ws=None) == 10
    assert call(wsb=ws_need - 1) == 10


def test_fused_host_validation(lib):
    """Checks that answer before the workspace size is computed (which asks the
    device for its SM count)."""
    f = lib.turnopd_fused_lmhead_fwd_bwd

    def call(hs=FAKE, Ws=FAKE, d_s=1024, ht=FAKE, Wt=FAKE, d_t=512, vocab=8192, T=64, mode=0, dh=FAKE, dW=None,
             tl=FAKE, loss=FAKE, ws=None, status=FAKE):
        return f(hs, Ws, d_s, ht, Wt, d_t, vocab, FAKE, FAKE, T, mode, dh, dW, tl, loss, ws, 1 << 30, status, None)

    assert call(Ws=None) == 1
    assert call(Wt=None) == 1
    assert call(loss=None) == 1
    assert call(status=None) == 1
    assert call(hs=None) == 1
    assert call(tl=None) == 1
    assert call(mode=1) == 6                                            # sampled mode is not fused
    assert call(d_s=1000) == 2                                          # d_s a multiple of 256
    assert call(d_s=128) == 2
    assert call(d_t=100) == 2                                           # d_t a multiple of 64
    assert call(d_s=65536 + 256) == 2
    assert call(vocab=0) == 2
    assert call(T=-1) == 2
    assert call(hs=ctypes.c_void_p(0x10008)) == 2                       # TMA operands 16-byte aligned
    assert call(dW=ctypes.c_void_p(0x10004)) == 2
    assert call() == 10                                                 # no workspace


def test_static_entry_rejects_oversize_batches(lib):
    f = lib.turnopd_loss_fwd_bwd_static
    T = 65536 + 1                                                       # TURNOPD_STATIC_MAX_TOKENS + 1
    assert f(FAKE, FAKE, 1, 1024, 1024, T, None, None, FAKE, FAKE, T, 0, None, 0, 0, FAKE, FAKE, FAKE,
             None) == 10


def test_selftest_wait_timeout_host_validation(lib):
    f = lib.turnopd_selftest_wait_timeout
    assert f(100, None, None) == 1                # TURNOPD_ERR_NULL
    assert f(0, FAKE, None) == 2                  # TURNOPD_ERR_SHAPE: no polls
    assert f((1 << 24) + 1, FAKE, None) == 2      # TURNOPD_ERR_SHAPE: beyond the cap


def declared_parameter_counts():
    """name -> number of parameters, from every prototype in the header."""
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    out = {}
    for m in re.finditer(r"^[A-Za-z_][\w \*]*?\b(turnopd_\w+)\s*\(([^;{]*?)\)\s*;", src, flags=re.M | re.S):
        params = m.group(2).strip()
        out[m.group(1)] = 0 if params in ("", "void") else params.count(",") + 1
    return out


def test_binding_argument_counts_match_header(lib):
    counts = declared_parameter_counts()
    assert "turnopd_vocab_shard_stats" in counts and "turnopd_loss_fwd_bwd" in counts
    checked = 0
    for name, n in counts.items():
        argtypes = getattr(lib, name).argtypes
        if argtypes is None:
            continue
        assert len(argtypes) == n, (name, len(argtypes), n)
        checked += 1
    assert checked >= 20
