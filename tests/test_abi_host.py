"""Host-side checks of the C ABI (no GPU needed).

The library must load and export every entry point include/retrace.h
declares; workspace sizing is pure host arithmetic; invalid arguments come back
as status codes before anything touches CUDA.
"""

import ctypes
import os
import re

import pytest

from paper_2608_29748_gb300 import build as libbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "retrace.h")

OK, INVALID, UNSUPPORTED, WORKSPACE = 0, 1, 2, 3
F32, BF16 = 0, 1


@pytest.fixture(scope="module")
def lib():
    path = libbuild.build()
    L = ctypes.CDLL(path)
    L.retrace_workspace_bytes.restype = ctypes.c_size_t
    L.retrace_workspace_bytes.argtypes = [ctypes.c_int] * 5
    L.retrace_last_error.restype = ctypes.c_char_p
    L.retrace_version.restype = ctypes.c_char_p
    return L


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(retrace_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_round_entry_points():
    names = declared_functions()
    for n in ("retrace_verify", "retrace_align_refine", "retrace_gate_fuse", "retrace_round",
              "retrace_workspace_bytes", "retrace_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_version_string(lib):
    assert b"sm_103a" in lib.retrace_version()


def test_workspace_bytes(lib):
    ws = lib.retrace_workspace_bytes
    assert ws(-1, 16, 10, 8, BF16) == 0
    assert ws(1, 16, 0, 8, BF16) == 0
    assert ws(1, 16, 10, 8, 7) == 0
    small = ws(1, 16, 151936, 2560, BF16)
    big = ws(256, 16, 151936, 4096, BF16)
    assert 0 < small < big
    assert big % 256 == 0
    # keys (8 B per row of K+1) + tickets + gate vector + compact r in bf16
    assert big >= 256 * 17 * 8 + 256 * 4 + 4096 * 4 + 256 * 15 * 4096 * 2
    assert ws(256, 16, 151936, 4096, F32) > big  # r stored in fp32 for fp32 workloads
    assert ws(0, 16, 10, 8, BF16) > 0  # empty batch: still a valid (tiny) workspace


def _verify(lib, logits=16, dtype=BF16, B=2, K=4, V=10, rs=10, bs=50, ws=None, ws_bytes=1 << 20, draft=16):
    P = ctypes.c_void_p
    return lib.retrace_verify(P(logits), dtype, B, K, V, ctypes.c_int64(rs), ctypes.c_int64(bs), P(draft),
                              P(16), P(16), P(16), None, P(ws) if ws else None, ctypes.c_size_t(ws_bytes), None)


def test_verify_argument_errors(lib):
    assert _verify(lib, logits=0) == INVALID
    assert _verify(lib, draft=0) == INVALID
    assert _verify(lib, dtype=9) == INVALID
    assert _verify(lib, V=0) == INVALID
    assert _verify(lib, rs=9) == INVALID  # row stride below V
    assert _verify(lib, bs=49) == INVALID  # batch stride below (K+1)*row_stride
    assert _verify(lib, K=5000, bs=10 ** 6) == UNSUPPORTED
    assert _verify(lib, ws=None) == WORKSPACE
    assert _verify(lib, ws=256 * 3, ws_bytes=8) == WORKSPACE
    assert _verify(lib, ws=256 * 3 + 8) == WORKSPACE  # misaligned workspace
    assert b"workspace" in lib.retrace_last_error()
    assert _verify(lib, B=0, logits=0, draft=0) == OK  # empty batch is a no-op


def test_conditioning_argument_errors(lib):
    P = ctypes.c_void_p
    f = ctypes.c_float(1.0)
    sz = ctypes.c_size_t(1 << 20)
    # K must be >= 1 for conditioning
    assert lib.retrace_align_refine(P(16), P(16), BF16, 2, 0, 8, P(16), P(16), f, P(16), P(16), P(256), sz, None) == INVALID
    assert lib.retrace_align_refine(None, P(16), BF16, 2, 4, 8, P(16), P(16), f, P(16), P(16), P(256), sz, None) == INVALID
    # e strides other than broadcast (0, 0) or dense (K*d, d)
    st = lib.retrace_gate_fuse(P(16), ctypes.c_int64(8), ctypes.c_int64(8), P(16), P(16), P(16), P(16), BF16,
                               2, 4, 8, P(16), P(256), sz, None)
    assert st == UNSUPPORTED
    assert b"strides" in lib.retrace_last_error()


def test_workspace_init_rejects_null(lib):
    lib.retrace_workspace_init.argtypes = [ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]
    assert lib.retrace_workspace_init(None, 128, None) == INVALID


def _round(lib, flags, Wc=16, Wv=16, Wg=16, B=0):
    """retrace_round with fake pointers; every case here returns before any
    CUDA call (argument checks, or B = 0)."""
    P, I64 = ctypes.c_void_p, ctypes.c_int64
    return lib.retrace_round(P(16), I64(10), I64(50), P(16), P(16), P(16), P(16), I64(0), I64(0),
                             P(Wc) if Wc else None, P(Wv) if Wv else None, P(Wg) if Wg else None,
                             ctypes.c_float(1.0), BF16, B, 4, 10, 8, P(16), P(16), P(16), None, None, P(16),
                             P(256), ctypes.c_size_t(1 << 20), ctypes.c_uint32(flags), None, None)


def test_round_flag_errors(lib):
    RAW, OVERWRITE, NONE, OVERLAP = 0x2, 0x4, 0x8, 0x1
    assert _round(lib, 0x100) == INVALID  # unknown bit
    assert b"flag" in lib.retrace_last_error()
    assert _round(lib, RAW | NONE) == INVALID  # two ablation variants
    assert _round(lib, OVERWRITE | RAW) == INVALID
    assert _round(lib, OVERLAP | RAW) == UNSUPPORTED  # the overlapped kernel runs the method only
    for flags in (0, RAW, OVERWRITE, NONE, OVERLAP):
        assert _round(lib, flags) == OK  # B = 0: nothing to do


def test_round_header_documents_the_flags():
    text = open(HEADER).read()
    for name, value in (("RETRACE_ROUND_OVERLAP", 0x1), ("RETRACE_COND_RAW", 0x2),
                        ("RETRACE_COND_OVERWRITE", 0x4), ("RETRACE_COND_NONE", 0x8)):
        m = re.search(r"#define\s+%s\s+(0x[0-9a-fA-F]+)u" % name, text)
        assert m and int(m.group(1), 16) == value, name


def _sampled(lib, T=1.0, k=20, p=0.95, B=2, K=4, V=100, dl=16, u=16, drs=100, dbs=400):
    """retrace_verify_sampled with fake pointers; the cases here return
    before any CUDA call."""
    P, I64 = ctypes.c_void_p, ctypes.c_int64
    return lib.retrace_verify_sampled(P(16), I64(V), I64((K + 1) * V), P(dl) if dl else None, I64(drs), I64(dbs),
                                      BF16, B, K, V, P(16), P(u) if u else None, ctypes.c_float(T), k,
                                      ctypes.c_float(p), P(16), P(16), P(16), P(256), ctypes.c_size_t(1 << 30), None)


def test_sampled_verification_argument_errors(lib):
    assert _sampled(lib, T=0.0) == INVALID
    assert _sampled(lib, T=float("inf")) == INVALID
    assert _sampled(lib, k=0) == INVALID
    assert _sampled(lib, k=65) == INVALID  # above the supported maximum
    assert _sampled(lib, k=20, V=10, drs=10, dbs=40) == INVALID  # top_k > V
    assert _sampled(lib, p=0.0) == INVALID
    assert _sampled(lib, p=1.5) == INVALID
    assert _sampled(lib, dl=0) == INVALID
    assert _sampled(lib, u=0) == INVALID
    assert _sampled(lib, drs=99) == INVALID  # drafter row stride below V
    assert _sampled(lib, dbs=399) == INVALID  # drafter batch stride below K * row stride
    assert _sampled(lib, B=0) == OK


def test_sampled_round_argument_errors(lib):
    P, I64, F = ctypes.c_void_p, ctypes.c_int64, ctypes.c_float

    def call(B=2, K=4, V=100, d=8, T=1.0, k=20, Wc=16, u=16, ebs=0, eps=0, ws_bytes=1 << 30):
        return lib.retrace_round_sampled(P(16), I64(V), I64((K + 1) * V), P(16), I64(V), I64(K * V), P(16),
                                         P(u) if u else None, F(T), k, F(0.95), P(16), P(16), P(16), I64(ebs),
                                         I64(eps), P(Wc) if Wc else None, P(16), P(16), F(1.0), BF16, B, K, V, d,
                                         P(16), P(16), P(16), None, P(16), P(256), ctypes.c_size_t(ws_bytes), None,
                                         None)

    assert call(Wc=0) == INVALID  # a NULL weight
    assert call(u=0) == INVALID
    assert call(T=-1.0) == INVALID
    assert call(k=65) == INVALID
    assert call(K=0) == INVALID
    assert call(d=0) == INVALID
    assert call(ebs=7, eps=3) == UNSUPPORTED  # e neither broadcast nor dense
    assert call(ws_bytes=64) == WORKSPACE  # workspace too small
    assert call(B=0) == OK


def test_wait_selftest_argument_errors(lib):
    P, U32 = ctypes.c_void_p, ctypes.c_uint32
    assert lib.retrace_wait_selftest(2, P(16), U32(1), P(256), ctypes.c_size_t(1 << 20), None) == INVALID
    assert lib.retrace_wait_selftest(0, None, U32(1), P(256), ctypes.c_size_t(1 << 20), None) == INVALID
    assert lib.retrace_wait_selftest(1, None, U32(1), P(256), ctypes.c_size_t(64), None) == WORKSPACE
    assert lib.retrace_wait_selftest(1, None, U32(1), P(100), ctypes.c_size_t(1 << 20), None) == WORKSPACE


def test_lowrank_round_argument_errors(lib):
    P, I64 = ctypes.c_void_p, ctypes.c_int64

    def call(B=2, P_=16, d=8, K=4):
        return lib.retrace_round_lowrank(P(16), I64(10), I64(50), P(16), P(16), P(16), P(16), P(P_) if P_ else None,
                                         P(16), P(16), P(16), P(16), ctypes.c_float(1.0), BF16, B, K, 10, d,
                                         P(16), P(16), P(16), None, None, P(16), P(256), ctypes.c_size_t(1 << 20),
                                         None, None)

    assert call(P_=0) == INVALID  # a NULL weight
    assert call(K=0) == INVALID
    assert call(d=0) == INVALID
    assert call(B=0) == OK


def _plan(lib, B, K, V, dtype=BF16, argmax=0):
    starts = (ctypes.c_int * 17)()
    lib.retrace_verify_plan.argtypes = [ctypes.c_int] * 5 + [ctypes.POINTER(ctypes.c_int)]
    n = lib.retrace_verify_plan(B, K, V, dtype, argmax, starts)
    return n, list(starts[: n + 1]) if n > 0 else []


def test_verify_schedule_plan(lib):
    """Windows of the windowed schedule: 4 rows, then half as long again each
    pass, a short remainder joining the last window; the automatic choice by
    batch size; target_argmax and short blocks keep one pass."""
    AUTO, FULL, WINDOWS = 0, 1, 2
    prev = lib.retrace_set_verify_schedule(AUTO)
    try:
        assert _plan(lib, 256, 16, 151936) == (3, [0, 4, 10, 17])      # 74 MiB per row of the batch
        assert _plan(lib, 64, 16, 151936) == (3, [0, 4, 10, 17])       # 18.5 MiB
        assert _plan(lib, 8, 16, 151936) == (1, [0, 17])               # 2.3 MiB: one pass
        assert _plan(lib, 256, 16, 151936, argmax=1) == (1, [0, 17])   # every row is an output
        assert lib.retrace_set_verify_schedule(WINDOWS) == AUTO
        assert _plan(lib, 8, 16, 151936) == (3, [0, 4, 10, 17])
        assert _plan(lib, 1, 4, 100) == (1, [0, 5])                    # K+1 = 5: one window
        assert _plan(lib, 1, 5, 100) == (2, [0, 4, 6])
        assert _plan(lib, 1, 6, 100) == (2, [0, 4, 7])
        assert _plan(lib, 1, 9, 100) == (2, [0, 4, 10])
        assert _plan(lib, 1, 11, 100) == (2, [0, 4, 12])               # 2 rows left < 6 / 2: joined
        assert _plan(lib, 1, 12, 100) == (3, [0, 4, 10, 13])
        n, s = _plan(lib, 2, 1024, 100)
        assert 2 <= n <= 16 and s[0] == 0 and s[-1] == 1025 and all(a < b for a, b in zip(s, s[1:]))
        assert _plan(lib, 0, 16, 100) == (1, [0, 17])
        assert _plan(lib, 1, 16, 0)[0] == -1 and _plan(lib, 1, 1025, 10)[0] == -1
        assert _plan(lib, 1, 16, 10, dtype=7)[0] == -1
        assert lib.retrace_set_verify_schedule(FULL) == WINDOWS
        assert _plan(lib, 256, 16, 151936) == (1, [0, 17])
        assert lib.retrace_set_verify_schedule(9) == -1
    finally:
        lib.retrace_set_verify_schedule(prev)


def test_workspace_holds_small_r_partials(lib):
    """At most 1024 conditioned rows (and the gate GEMM's work tiles within 256
    CTAs) the workspace also holds the split partials of the small-R GEMMs:
    256 CTAs x 128 weight rows x min(256, rows rounded to 16) fp32."""
    ws = lib.retrace_workspace_bytes
    for B, K, d in ((1, 16, 2560), (8, 16, 4096), (64, 16, 2560), (64, 17, 4096)):
        rows = (B * (K - 1) + 15) // 16 * 16
        part = 256 * 128 * min(256, rows) * 4
        assert ws(B, K, 1000, d, BF16) >= part
    small = ws(64, 17, 1000, 4096, BF16)   # 1024 rows: partials of 32 MiB
    large = ws(65, 17, 1000, 4096, BF16)   # 1040 rows: the CTA-pair path, 4 MiB of split-tile halves
    assert (32 - 4 - 1) << 20 < small - large < (32 - 4) << 20
    # fp32 takes the FFMA path: neither partial region
    assert ws(65, 17, 1000, 4096, F32) < ws(64, 17, 1000, 4096, F32) - (30 << 20)


def test_workspace_holds_pair_split_halves(lib):
    """Beyond the small-R path (bf16, d a multiple of 256) the workspace holds
    the K halves of the CTA-pair kernel's split gate tiles: 8 tiles x 2 halves
    x 2 CTAs x 128 rows x 256 fp32 columns, and their tickets in the sync area."""
    ws = lib.retrace_workspace_bytes
    split = 8 * 2 * 2 * 128 * 256 * 4
    for B, K, d in ((65, 17, 4096), (256, 16, 4096), (128, 16, 2560 + 256)):
        rows = B * (K - 1)
        # r, apack, epack (bf16) and the row map come on top of the split halves
        assert ws(B, K, 1000, d, BF16) > split + rows * d * 2 * 4
    # d not a multiple of 256 takes the FFMA path, without split halves: from
    # d = 4096 to 4224 the d-sized buffers grow by half as much as from 3840 to
    # 4096, and the split region goes
    a, b, c = (ws(256, 16, 1000, dd, BF16) for dd in (3840, 4096, 4224))
    assert abs((c - b) - ((b - a) // 2 - split)) <= 4096
