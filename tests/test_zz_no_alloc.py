"""retrace_verify_noalloc checked against retrace_verify, through the C ABI.

retrace_verify_noalloc is for callers that are handed only their input and
output buffers and cannot allocate device memory (a custom operator whose host
framework owns all device allocations, a serving loop that reserved its
memory budget up front).  It keeps its scratch in a fixed array inside the
library instead of a caller workspace, and must give exactly the results of
retrace_verify, whose outputs are all integers: the comparison is bit-exact.

The file name makes pytest collect it after every other test file, so a run
that stops at the first failure has run everything else before this.
"""

import ctypes

import pytest
import torch

from paper_2608_29748_gb300.workloads import plant_prefix

pytestmark = pytest.mark.gpu

SCRATCH_LIMIT = 65536  # RETRACE_NOALLOC_SCRATCH_BYTES in include/retrace.h


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    P, I, I64 = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64
    fn = binding.lib.retrace_verify_noalloc
    fn.argtypes = [P, I, I, I, I, I64, I64, P, P, P, P, P, P]
    fn.restype = I
    return binding


def case(B, K, V, dtype, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    logits = torch.randn((B, K + 1, V), generator=g, device="cuda").to(dtype)
    draft = torch.randint(0, V, (B, K), generator=g, device="cuda", dtype=torch.int64)
    a = torch.randint(0, K + 1, (B,), generator=g, device="cuda")
    plant_prefix(logits, draft, a, ties=True)
    return logits, draft.to(torch.int32)


def outputs(B, K):
    return [torch.full(s, -9, dtype=torch.int32, device="cuda") for s in ((B,), (B, K + 1), (B,), (B, K + 1))]


def call_noalloc(rt, logits, draft):
    B, K1, V = logits.shape
    acc, com, bon, targ = outputs(B, K1 - 1)
    code = rt.RETRACE_BF16 if logits.dtype == torch.bfloat16 else rt.RETRACE_F32
    st = rt.lib.retrace_verify_noalloc(logits.data_ptr(), code, B, K1 - 1, V, logits.stride(1), logits.stride(0),
                                       draft.data_ptr(), acc.data_ptr(), com.data_ptr(), bon.data_ptr(),
                                       targ.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == 0, rt.lib.retrace_last_error().decode()
    return acc, com, bon, targ


def call_workspace_version(rt, logits, draft):
    B, K1, V = logits.shape
    acc, com, bon, targ = outputs(B, K1 - 1)
    ws = rt.Workspace(B, K1 - 1, V, 8, logits.dtype)
    rt.retrace_verify(logits, draft, acc, com, bon, ws, target_argmax=targ)
    return acc, com, bon, targ


def test_noalloc_matches_workspace_verify_on_consecutive_calls(rt):
    # Different shapes back to back: whatever one call leaves in the shared
    # array must not leak into the next.
    cases = [case(64, 16, 151936, torch.bfloat16, seed=1), case(5, 7, 3001, torch.float32, seed=2),
             case(256, 16, 4099, torch.bfloat16, seed=3)]
    for logits, draft in cases + cases[:1]:
        got = call_noalloc(rt, logits, draft)
        want = call_workspace_version(rt, logits, draft)
        torch.cuda.synchronize()
        for name, a, b in zip(("accept_len", "committed", "bonus", "target_argmax"), got, want):
            assert torch.equal(a, b), name


def test_noalloc_without_argmax_output_matches_the_windowed_schedule(rt):
    """With target_argmax NULL at the serving shape (B = 256, K = 16,
    V = 151936, bf16), retrace_verify with a workspace verifies in row
    windows while retrace_verify_noalloc, which has no live lists, reads every
    row in one pass.  The integer outputs must still agree bit for bit, on two
    calls in a row."""
    B, K, V = 256, 16, 151936  # 256 * 17 keys + 256 counters: 35,840 bytes of scratch
    assert len(rt.retrace_verify_plan(B, K, V, torch.bfloat16)) > 2  # the workspace path is windowed
    logits, draft = case(B, K, V, torch.bfloat16, seed=5)
    code = rt.RETRACE_BF16
    stream = torch.cuda.current_stream().cuda_stream
    ws = rt.Workspace(B, K, V, 8, logits.dtype)
    for _ in range(2):
        got = outputs(B, K)[:3]
        st = rt.lib.retrace_verify_noalloc(logits.data_ptr(), code, B, K, V, logits.stride(1), logits.stride(0),
                                           draft.data_ptr(), got[0].data_ptr(), got[1].data_ptr(),
                                           got[2].data_ptr(), None, stream)
        assert st == 0, rt.lib.retrace_last_error().decode()
        want = outputs(B, K)[:3]
        rt.retrace_verify(logits, draft, want[0], want[1], want[2], ws)  # no target_argmax: windowed
        torch.cuda.synchronize()
        for name, a, b in zip(("accept_len", "committed", "bonus"), got, want):
            assert torch.equal(a, b), name


def test_noalloc_rejects_batches_beyond_the_fixed_scratch(rt):
    B, K, V = 512, 16, 64  # 512 * 17 keys of 8 bytes = 69632 bytes > 65536
    logits, draft = case(B, K, V, torch.bfloat16, seed=4)
    acc, com, bon, targ = outputs(B, K)
    st = rt.lib.retrace_verify_noalloc(logits.data_ptr(), rt.RETRACE_BF16, B, K, V, logits.stride(1),
                                       logits.stride(0), draft.data_ptr(), acc.data_ptr(), com.data_ptr(),
                                       bon.data_ptr(), None, torch.cuda.current_stream().cuda_stream)
    assert st == 2  # RETRACE_ERR_UNSUPPORTED
    msg = rt.lib.retrace_last_error().decode()
    assert "too large" in msg and str(SCRATCH_LIMIT) in msg
    torch.cuda.synchronize()
    assert int(acc.min()) == -9  # nothing was written
