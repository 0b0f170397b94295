"""Thin ctypes binding over libretrace (the C ABI in include/retrace.h).

Argument marshalling only: every step of the round runs in the library's CUDA
kernels.  Tensors are torch CUDA tensors used as device buffers; the functions
carry the C entry points' names.  If the library has not been built the
import fails loudly -- there is no fallback path.
"""

from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

RETRACE_F32 = 0
RETRACE_BF16 = 1

_STATUS = {
    0: "RETRACE_OK",
    1: "RETRACE_ERR_INVALID_ARG",
    2: "RETRACE_ERR_UNSUPPORTED",
    3: "RETRACE_ERR_WORKSPACE",
    4: "RETRACE_ERR_CUDA",
    5: "RETRACE_ERR_DEVICE",
}


class RetraceError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


def _load() -> ctypes.CDLL:
    path = _build.LIB_PATH
    if not os.path.exists(path):
        raise ImportError(
            f"libretrace.so is not built ({path}); run `python -m paper_2608_29748_gb300.build` "
            "or __graft_entry__.build() first"
        )
    lib = ctypes.CDLL(path)
    P, I, I64, SZ, F = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t, ctypes.c_float
    lib.retrace_last_error.restype = ctypes.c_char_p
    lib.retrace_version.restype = ctypes.c_char_p
    lib.retrace_workspace_bytes.argtypes = [I, I, I, I, I]
    lib.retrace_workspace_bytes.restype = SZ
    lib.retrace_workspace_init.argtypes = [P, SZ, P]
    lib.retrace_workspace_check.argtypes = [P, SZ, ctypes.POINTER(ctypes.c_uint32), P]
    lib.retrace_verify.argtypes = [P, I, I, I, I, I64, I64, P, P, P, P, P, P, SZ, P]
    lib.retrace_align_refine.argtypes = [P, P, I, I, I, I, P, P, F, P, P, P, SZ, P]
    lib.retrace_gate_fuse.argtypes = [P, I64, I64, P, P, P, P, I, I, I, I, P, P, SZ, P]
    lib.retrace_round.argtypes = [P, I64, I64, P, P, P, P, I64, I64, P, P, P, F, I, I, I, I, I,
                                  P, P, P, P, P, P, P, SZ, ctypes.c_uint32, P, P]
    lib.retrace_round_lowrank.argtypes = [P, I64, I64, P, P, P, P, P, P, P, P, P, F, I, I, I, I, I,
                                          P, P, P, P, P, P, P, SZ, P, P]
    lib.retrace_verify_sampled.argtypes = [P, I64, I64, P, I64, I64, I, I, I, I, P, P, F, I, F, P, P, P, P, SZ, P]
    lib.retrace_wait_selftest.argtypes = [I, P, ctypes.c_uint32, P, SZ, P]
    lib.retrace_set_verify_schedule.argtypes = [I]
    lib.retrace_verify_plan.argtypes = [I, I, I, I, I, ctypes.POINTER(ctypes.c_int)]
    lib.retrace_round_sampled.argtypes = [P, I64, I64, P, I64, I64, P, P, F, I, F, P, P, P, I64, I64, P, P, P, F,
                                          I, I, I, I, I, P, P, P, P, P, P, SZ, P, P]
    for name in ("retrace_workspace_init", "retrace_workspace_check", "retrace_verify",
                 "retrace_align_refine", "retrace_gate_fuse", "retrace_round", "retrace_round_lowrank",
                 "retrace_verify_sampled", "retrace_round_sampled", "retrace_wait_selftest",
                 "retrace_set_verify_schedule", "retrace_verify_plan"):
        getattr(lib, name).restype = I
    return lib


lib = _load()


def _check(status: int) -> None:
    if status != 0:
        raise RetraceError(status, lib.retrace_last_error().decode())


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return RETRACE_BF16
    if t.dtype == torch.float32:
        return RETRACE_F32
    raise TypeError(f"unsupported floating dtype {t.dtype}")


def _ptr(t):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libretrace takes CUDA tensors")
    return t.data_ptr()


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def retrace_workspace_bytes(B: int, K: int, V: int, d: int, dtype: torch.dtype) -> int:
    code = RETRACE_BF16 if dtype == torch.bfloat16 else RETRACE_F32
    return int(lib.retrace_workspace_bytes(B, K, V, d, code))


class Workspace:
    """Caller-owned device workspace sized for (B, K, V, d, dtype), zeroed once."""

    def __init__(self, B, K, V, d, dtype, device=None, stream=None):
        self.nbytes = retrace_workspace_bytes(B, K, V, d, dtype)
        if self.nbytes == 0:
            raise ValueError("invalid workspace shape")
        self.buf = torch.empty(self.nbytes + 256, dtype=torch.uint8, device=device or "cuda")
        base = self.buf.data_ptr()
        self.ptr = (base + 255) // 256 * 256
        retrace_workspace_init(self, stream)

    def check(self, stream=None) -> int:
        return retrace_workspace_check(self, stream)


def retrace_workspace_init(ws: Workspace, stream=None) -> None:
    _check(lib.retrace_workspace_init(ws.ptr, ws.nbytes, _stream(stream)))


def retrace_workspace_check(ws: Workspace, stream=None) -> int:
    flags = ctypes.c_uint32(0)
    st = lib.retrace_workspace_check(ws.ptr, ws.nbytes, ctypes.byref(flags), _stream(stream))
    if st not in (0, 5):
        _check(st)
    return int(flags.value)


def _int32(t: torch.Tensor, name: str) -> None:
    if t.dtype != torch.int32:
        raise TypeError(f"{name} must be int32")


def retrace_verify(logits, draft, accept_len, committed, bonus, ws, target_argmax=None, stream=None):
    """Greedy verification (see include/retrace.h).  logits [B, K+1, V], last dim contiguous."""
    B, K1, V = logits.shape
    if logits.stride(2) != 1:
        raise ValueError("logits: vocabulary dimension must be contiguous")
    for t, n in ((draft, "draft"), (accept_len, "accept_len"), (committed, "committed"), (bonus, "bonus")):
        _int32(t, n)
    _check(lib.retrace_verify(_ptr(logits), _dtype_code(logits), B, K1 - 1, V, logits.stride(1),
                              logits.stride(0), _ptr(draft), _ptr(accept_len), _ptr(committed),
                              _ptr(bonus), _ptr(target_argmax), ws.ptr, ws.nbytes, _stream(stream)))


def retrace_align_refine(hD, hT, accept_len, Wc, beta, r_out, n_out, ws, stream=None):
    """Alignment + target-aware correction: r_out [B, K, d], n_out [B]."""
    B, K, d = hD.shape
    for t in (hD, hT, Wc, r_out):
        if not t.is_contiguous():
            raise ValueError("hD, hT, Wc and r_out must be contiguous")
    _check(lib.retrace_align_refine(_ptr(hD), _ptr(hT), _dtype_code(hD), B, K, d, _ptr(accept_len),
                                    _ptr(Wc), float(beta), _ptr(r_out), _ptr(n_out), ws.ptr,
                                    ws.nbytes, _stream(stream)))


def _e_strides(e: torch.Tensor, B: int, K: int, d: int):
    if e.dim() == 1:
        return 0, 0
    if e.shape != (B, K, d) or not e.is_contiguous():
        raise ValueError("e must be a [d] vector or a contiguous [B, K, d] tensor")
    return K * d, d


def retrace_gate_fuse(e, r, n, Wv, Wg, e_out, ws, stream=None):
    """Gated residual conditioning: e_out [B, K, d]."""
    B, K, d = r.shape
    ebs, eps = _e_strides(e, B, K, d)
    _check(lib.retrace_gate_fuse(_ptr(e), ebs, eps, _ptr(r), _ptr(n), _ptr(Wv), _ptr(Wg),
                                 _dtype_code(r), B, K, d, _ptr(e_out), ws.ptr, ws.nbytes,
                                 _stream(stream)))


# retrace_round flags (include/retrace.h)
ROUND_OVERLAP = 0x1
COND_RAW = 0x2
COND_OVERWRITE = 0x4
COND_NONE = 0x8


def retrace_round(logits, draft, hD, hT, e, Wc, Wv, Wg, beta, accept_len, committed, bonus, e_out,
                  ws, n_out=None, target_argmax=None, flags=0, phase_events=None, stream=None):
    """One round on one stream (see include/retrace.h); `flags` selects the
    overlapped kernel or an ablation variant."""
    B, K1, V = logits.shape
    K = K1 - 1
    d = hD.shape[2]
    if logits.stride(2) != 1:
        raise ValueError("logits: vocabulary dimension must be contiguous")
    ebs, eps = _e_strides(e, B, K, d)
    ev = None
    if phase_events is not None:
        ev = (ctypes.c_void_p * 4)(*[x._as_parameter_.value for x in phase_events])
    _check(lib.retrace_round(_ptr(logits), logits.stride(1), logits.stride(0), _ptr(draft), _ptr(hD),
                             _ptr(hT), _ptr(e), ebs, eps, _ptr(Wc), _ptr(Wv), _ptr(Wg), float(beta),
                             _dtype_code(logits), B, K, V, d, _ptr(accept_len), _ptr(committed),
                             _ptr(bonus), _ptr(target_argmax), _ptr(n_out), _ptr(e_out), ws.ptr,
                             ws.nbytes, int(flags),
                             ctypes.cast(ev, ctypes.c_void_p) if ev is not None else None,
                             _stream(stream)))


def retrace_verify_sampled(target_logits, draft_logits, draft, uniforms, temperature, top_k, top_p, accept_len,
                           committed, bonus, ws, stream=None):
    """Speculative sampling of one block per sequence (see include/retrace.h)."""
    _check_sampled(target_logits, draft_logits, uniforms)
    B, K1, V = target_logits.shape
    K = K1 - 1
    for t, name in ((draft, "draft"), (accept_len, "accept_len"), (committed, "committed"), (bonus, "bonus")):
        _int32(t, name)
    _check(lib.retrace_verify_sampled(_ptr(target_logits), target_logits.stride(1), target_logits.stride(0),
                                      _ptr(draft_logits), draft_logits.stride(1), draft_logits.stride(0),
                                      _dtype_code(target_logits), B, K, V, _ptr(draft), _ptr(uniforms),
                                      float(temperature), int(top_k), float(top_p), _ptr(accept_len),
                                      _ptr(committed), _ptr(bonus), ws.ptr, ws.nbytes, _stream(stream)))


def _check_sampled(target_logits, draft_logits, uniforms):
    B, K1, V = target_logits.shape
    K = K1 - 1
    if target_logits.stride(2) != 1 or draft_logits.stride(2) != 1:
        raise ValueError("logits: vocabulary dimension must be contiguous")
    if tuple(draft_logits.shape) != (B, K, V) or draft_logits.dtype != target_logits.dtype:
        raise ValueError("draft_logits must be [B, K, V] of the target logits' dtype")
    if uniforms.dtype != torch.float32 or tuple(uniforms.shape) != (B, K1) or not uniforms.is_contiguous():
        raise ValueError("uniforms must be contiguous float32 [B, K+1]")


def retrace_round_sampled(target_logits, draft_logits, draft, uniforms, temperature, top_k, top_p, hD, hT, e, Wc,
                          Wv, Wg, beta, accept_len, committed, bonus, e_out, ws, n_out=None, phase_events=None,
                          stream=None):
    """One round with sampled verification (see include/retrace.h)."""
    _check_sampled(target_logits, draft_logits, uniforms)
    B, K1, V = target_logits.shape
    K = K1 - 1
    d = hD.shape[2]
    for t, name in ((draft, "draft"), (accept_len, "accept_len"), (committed, "committed"), (bonus, "bonus")):
        _int32(t, name)
    ebs, eps = _e_strides(e, B, K, d)
    ev = None
    if phase_events is not None:
        ev = (ctypes.c_void_p * 4)(*[x._as_parameter_.value for x in phase_events])
    _check(lib.retrace_round_sampled(_ptr(target_logits), target_logits.stride(1), target_logits.stride(0),
                                     _ptr(draft_logits), draft_logits.stride(1), draft_logits.stride(0), _ptr(draft),
                                     _ptr(uniforms), float(temperature), int(top_k), float(top_p), _ptr(hD), _ptr(hT),
                                     _ptr(e), ebs, eps, _ptr(Wc), _ptr(Wv), _ptr(Wg), float(beta),
                                     _dtype_code(target_logits), B, K, V, d, _ptr(accept_len), _ptr(committed),
                                     _ptr(bonus), _ptr(n_out), _ptr(e_out), ws.ptr, ws.nbytes,
                                     ctypes.cast(ev, ctypes.c_void_p) if ev is not None else None,
                                     _stream(stream)))


def retrace_round_lowrank(logits, draft, hD, hT, e, P, Bc, Ac, Wv, Wg, beta, accept_len, committed, bonus,
                          e_out, ws, n_out=None, target_argmax=None, phase_events=None, stream=None):
    """One round with the low-rank conditioning path (see include/retrace.h)."""
    B, K1, V = logits.shape
    K = K1 - 1
    d = hD.shape[2]
    if logits.stride(2) != 1:
        raise ValueError("logits: vocabulary dimension must be contiguous")
    if e.dim() != 1:
        raise ValueError("e: the low-rank path takes one broadcast vector [d]")
    ev = None
    if phase_events is not None:
        ev = (ctypes.c_void_p * 4)(*[x._as_parameter_.value for x in phase_events])
    _check(lib.retrace_round_lowrank(_ptr(logits), logits.stride(1), logits.stride(0), _ptr(draft), _ptr(hD),
                                     _ptr(hT), _ptr(e), _ptr(P), _ptr(Bc), _ptr(Ac), _ptr(Wv), _ptr(Wg),
                                     float(beta), _dtype_code(logits), B, K, V, d, _ptr(accept_len),
                                     _ptr(committed), _ptr(bonus), _ptr(target_argmax), _ptr(n_out), _ptr(e_out),
                                     ws.ptr, ws.nbytes,
                                     ctypes.cast(ev, ctypes.c_void_p) if ev is not None else None,
                                     _stream(stream)))


def retrace_wait_selftest(kind, flag, target, ws, stream=None):
    """Runs the kernels' bounded wait on a caller-controlled condition (see include/retrace.h)."""
    if flag is not None and flag.dtype != torch.int32:
        raise TypeError("flag must be an int32 device tensor")
    _check(lib.retrace_wait_selftest(int(kind), _ptr(flag), int(target), ws.ptr, ws.nbytes, _stream(stream)))


class RoundBuffers:
    """Device outputs of one round for a (B, K, d) shape."""

    def __init__(self, B, K, d, dtype, device="cuda"):
        self.accept_len = torch.empty(B, dtype=torch.int32, device=device)
        self.committed = torch.empty(B, K + 1, dtype=torch.int32, device=device)
        self.bonus = torch.empty(B, dtype=torch.int32, device=device)
        self.n = torch.empty(B, dtype=torch.int32, device=device)
        self.e_out = torch.empty(B, K, d, dtype=dtype, device=device)


def run_round(x: dict, ws: Workspace, out: RoundBuffers | None = None, target_argmax=None,
              flags=0, phase_events=None, stream=None) -> RoundBuffers:
    """retrace_round over a dict of device tensors (keys as in workloads.make_round_inputs)."""
    logits = x["logits"]
    B, K1, _ = logits.shape
    d = x["hD"].shape[2]
    if out is None:
        out = RoundBuffers(B, K1 - 1, d, logits.dtype, logits.device)
    retrace_round(logits, x["draft"], x["hD"], x["hT"], x["e"], x["Wc"], x["Wv"], x["Wg"], x["beta"],
                  out.accept_len, out.committed, out.bonus, out.e_out, ws, n_out=out.n,
                  target_argmax=target_argmax, flags=flags, phase_events=phase_events, stream=stream)
    return out


def version() -> str:
    return lib.retrace_version().decode()


VERIFY_AUTO, VERIFY_FULL, VERIFY_WINDOWS = 0, 1, 2


def retrace_verify_plan(B: int, K: int, V: int, dtype: torch.dtype, target_argmax: bool = False) -> list[int]:
    """Window boundaries greedy verification takes for this shape under the
    current schedule ([0, K+1] for the one-pass schedule)."""
    starts = (ctypes.c_int * 17)()
    code = RETRACE_BF16 if dtype == torch.bfloat16 else RETRACE_F32 if dtype == torch.float32 else -1
    n = lib.retrace_verify_plan(B, K, V, code, int(bool(target_argmax)), starts)
    if n < 1:
        raise RetraceError(1, "invalid shape or dtype for retrace_verify_plan")
    return list(starts[: n + 1])


def retrace_set_verify_schedule(mode: int) -> int:
    """Selects the greedy verification schedule (VERIFY_AUTO / VERIFY_FULL /
    VERIFY_WINDOWS); returns the previous one."""
    prev = lib.retrace_set_verify_schedule(int(mode))
    if prev < 0:
        raise RetraceError(1, f"unknown verification schedule {mode}")
    return prev


def run_round_lowrank(x: dict, w: dict, ws: Workspace, out: RoundBuffers | None = None, target_argmax=None,
                      phase_events=None, stream=None) -> RoundBuffers:
    """retrace_round_lowrank over the round inputs ``x`` and low-rank weights ``w``
    (keys as in workloads.make_round_inputs / make_lowrank_weights)."""
    logits = x["logits"]
    B, K1, _ = logits.shape
    d = x["hD"].shape[2]
    if out is None:
        out = RoundBuffers(B, K1 - 1, d, logits.dtype, logits.device)
    retrace_round_lowrank(logits, x["draft"], x["hD"], x["hT"], x["e"], w["P"], w["Bc"], w["Ac"], w["Wv_lr"],
                          w["Wg_lr"], x["beta"], out.accept_len, out.committed, out.bonus, out.e_out, ws,
                          n_out=out.n, target_argmax=target_argmax, phase_events=phase_events, stream=stream)
    return out


def run_round_sampled(x: dict, s: dict, ws: Workspace, out: RoundBuffers | None = None, phase_events=None,
                      stream=None) -> RoundBuffers:
    """retrace_round_sampled over the round inputs ``x`` (its logits are the
    target's) and the sampling inputs ``s`` (keys as in
    workloads.make_sampled_inputs; its draft tokens replace x["draft"])."""
    logits = x["logits"]
    B, K1, _ = logits.shape
    d = x["hD"].shape[2]
    if out is None:
        out = RoundBuffers(B, K1 - 1, d, logits.dtype, logits.device)
    retrace_round_sampled(logits, s["draft_logits"], s["draft"], s["uniforms"], s["temperature"], s["top_k"],
                          s["top_p"], x["hD"], x["hT"], x["e"], x["Wc"], x["Wv"], x["Wg"], x["beta"], out.accept_len,
                          out.committed, out.bonus, out.e_out, ws, n_out=out.n, phase_events=phase_events,
                          stream=stream)
    return out
