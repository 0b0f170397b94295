"""GPU parity of the windowed verification schedule vs the oracle.

Without target_argmax the outputs depend only on rows 0..A_b of every
sequence; the windowed schedule reads rows in passes over windows of rows,
each pass only for the sequences whose draft tokens matched every earlier
row, through live lists in the workspace.  Its results must equal the
oracle's bit for bit on every shape the one-pass schedule is tested on
(vector and element-wise paths, ragged row tails, every acceptance pattern),
call after call on one workspace (the live counters, keys and tickets must
be left clean), inside CUDA graphs, and inside the fused round.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import host_f64, host_int
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, plant_prefix

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


@pytest.fixture
def windows(rt):
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_WINDOWS)
    yield
    rt.retrace_set_verify_schedule(prev)


def verify_no_argmax(rt, logits, draft, ws=None):
    B, K1, V = logits.shape
    K = K1 - 1
    if ws is None:
        ws = rt.Workspace(B, K, V, 8, logits.dtype)
    acc = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    com = torch.full((B, K + 1), -7, dtype=torch.int32, device="cuda")
    bon = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    rt.retrace_verify(logits, draft, acc, com, bon, ws)
    torch.cuda.synchronize()
    return acc, com, bon


def check(rt, logits, draft, ws=None):
    acc, com, bon = verify_no_argmax(rt, logits, draft, ws)
    want = oracle.verify(host_f64(logits), host_int(draft))
    np.testing.assert_array_equal(host_int(acc), want["accept_len"])
    np.testing.assert_array_equal(host_int(com), want["committed"])
    np.testing.assert_array_equal(host_int(bon), want["bonus"])
    return want


def random_case(B, K, V, dtype, seed, ties=False, accept=None):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    logits = torch.randn((B, K + 1, V), generator=g, device="cuda").to(dtype)
    draft = torch.randint(0, V, (B, K), generator=g, device="cuda", dtype=torch.int64)
    a = torch.randint(0, K + 1, (B,), generator=g, device="cuda") if accept is None else accept.cuda()
    plant_prefix(logits, draft, a, ties=ties)
    return logits, draft.to(torch.int32)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize(
    "B,K,V",
    [(1, 0, 8), (3, 0, 4096), (1, 1, 8), (2, 1, 16), (3, 3, 8), (5, 16, 1024), (1, 16, 1032),
     (37, 5, 4104), (4, 40, 3008), (2, 16, 100008), (1, 16, 151936), (300, 16, 4096), (3, 7, 151944)],
)
def test_windows_shapes(rt, windows, B, K, V, dtype):
    logits, draft = random_case(B, K, V, dtype, seed=B * 1000 + K * 10 + V, ties=V > 16)
    check(rt, logits, draft)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V", [1001, 4099, 151939])
def test_windows_strided_ragged_rows(rt, windows, dtype, V):
    """Aligned row stride, V not a multiple of the 16-byte vector: the last
    elements of each row are read one by one."""
    B, K = 9, 6
    Vp = (V + 63) // 64 * 64
    big, draft = random_case(B, K, Vp, dtype, seed=V)
    logits = big[:, :, :V]
    draft = torch.where(draft >= V, draft % V, draft)
    for b in range(B):  # a maximum in the ragged tail of some rows
        logits[b, b % (K + 1), V - 1] = 50.0
    check(rt, logits, draft)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("pad", [3, 8])
def test_windows_strided_logits(rt, windows, dtype, pad):
    """Row stride V + pad: pad 3 takes the element-wise path."""
    B, K, V = 5, 16, 5000
    big, draft = random_case(B, K + 2, V + pad, dtype, seed=pad)
    logits = big[:, : K + 1, :V]
    check(rt, logits, draft[:, :K].contiguous())


@pytest.mark.parametrize("K", [4, 5, 6, 7, 8, 9, 40, 300])
def test_windows_pass_boundaries(rt, windows, K):
    """Every accepted length from 0 to K, across the window boundaries, with
    the last window merged or not (K + 1 = 5 .. 10 rows) and with widened
    windows for long blocks."""
    B, V = K + 1, 2048
    logits, draft = random_case(B, K, V, torch.bfloat16, seed=K, accept=torch.arange(B))
    want = check(rt, logits, draft)
    assert list(want["accept_len"]) == list(range(B))


@pytest.mark.parametrize("cfg_id", [1, 2, 3, 4, 5])
def test_windows_workloads(rt, windows, cfg_id):
    x = make_round_inputs(CONFIGS[cfg_id], device="cuda")
    want = check(rt, x["logits"], x["draft"])
    assert np.array_equal(want["accept_len"], x["planted_prefix"].cpu().numpy())


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_windows_all_accepted_and_all_rejected(rt, windows, dtype):
    """Every sequence is read to row K (bonus row), or stops in the first window."""
    B, K, V = 64, 16, 20000
    for a in (torch.full((B,), K), torch.zeros(B, dtype=torch.int64)):
        logits, draft = random_case(B, K, V, dtype, seed=int(a[0]), accept=a)
        want = check(rt, logits, draft)
        assert np.all(want["accept_len"] == int(a[0]))


def test_windows_dense_ties_lowest_index(rt, windows):
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    B, K, V = 6, 8, 151936
    vals = torch.tensor([-1.0, 0.0, 0.5, 1.0], device="cuda")
    logits = vals[torch.randint(0, 4, (B, K + 1, V), generator=g, device="cuda")].to(torch.bfloat16)
    # draft = the first maximum index of each row: every row matches, all rows are read
    targ = oracle.target_argmax(host_f64(logits))
    draft = torch.from_numpy(targ[:, :K].astype(np.int32)).cuda()
    draft[2, 3] += 1  # one sequence stops at row 3 (a later tie index does not match)
    want = check(rt, logits, draft)
    assert want["accept_len"][2] == 3 and want["accept_len"][0] == K


def test_windows_workspace_left_clean(rt, windows):
    """Calls with changing shapes and acceptance patterns on one workspace,
    interleaved with one-pass calls: every result equals the oracle, so no
    queue slot, part counter or key is left behind by either schedule."""
    ws = rt.Workspace(256, 16, 151936, 8, torch.bfloat16)
    cases = [random_case(256, 16, 20000, torch.bfloat16, seed=s, ties=True) for s in (1, 2)]
    cases.append(random_case(3, 5, 1000, torch.bfloat16, seed=9))
    cases.append(random_case(256, 16, 20000, torch.bfloat16, seed=3, accept=torch.full((256,), 16)))
    wants = [oracle.verify(host_f64(l), host_int(d)) for l, d in cases]
    for it in range(12):
        c = it % len(cases)
        if it % 3 == 2:
            rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
        acc, com, bon = verify_no_argmax(rt, *cases[c], ws=ws)
        rt.retrace_set_verify_schedule(rt.VERIFY_WINDOWS)
        np.testing.assert_array_equal(host_int(acc), wants[c]["accept_len"])
        np.testing.assert_array_equal(host_int(com), wants[c]["committed"])
        np.testing.assert_array_equal(host_int(bon), wants[c]["bonus"])
    assert ws.check() == 0


def test_windows_batch_limit(rt):
    """The default schedule verifies in row windows up to B = 2048 sequences
    (each CTA keeps the live lists and decisions of the whole batch in shared
    memory) and in one pass above that; both against the oracle, on the
    smallest rows that still make one row of the batch 16 MiB."""
    K, V = 8, 4104
    for B, windowed in ((2048, True), (2049, False)):
        assert (len(rt.retrace_verify_plan(B, K, V, torch.bfloat16)) > 2) == windowed
        logits, draft = random_case(B, K, V, torch.bfloat16, seed=B, ties=True)
        check(rt, logits, draft)


def test_windows_in_cuda_graph(rt, windows):
    """Captured once, replayed on new logits written into the same buffer."""
    B, K, V = 128, 16, 30000
    cases = [random_case(B, K, V, torch.bfloat16, seed=s) for s in (11, 12, 13)]
    logits = cases[0][0].clone()
    draft = cases[0][1].clone()
    ws = rt.Workspace(B, K, V, 8, torch.bfloat16)
    acc = torch.empty((B,), dtype=torch.int32, device="cuda")
    com = torch.empty((B, K + 1), dtype=torch.int32, device="cuda")
    bon = torch.empty((B,), dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        rt.retrace_verify(logits, draft, acc, com, bon, ws, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        rt.retrace_verify(logits, draft, acc, com, bon, ws, stream=s)
    for l, d in cases[1:] + cases[:1]:
        logits.copy_(l)
        draft.copy_(d)
        g.replay()
        torch.cuda.synchronize()
        want = oracle.verify(host_f64(l), host_int(d))
        np.testing.assert_array_equal(host_int(acc), want["accept_len"])
        np.testing.assert_array_equal(host_int(com), want["committed"])
    assert ws.check() == 0


def test_schedule_setter(rt):
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    assert rt.retrace_set_verify_schedule(rt.VERIFY_AUTO) == rt.VERIFY_FULL
    with pytest.raises(rt.RetraceError):
        rt.retrace_set_verify_schedule(7)
    assert rt.retrace_set_verify_schedule(prev) == rt.VERIFY_AUTO


@pytest.mark.parametrize("cfg_id", [1, 3, 4])
@pytest.mark.parametrize("flags", ["default", "raw", "overwrite", "none"])
def test_round_outputs_identical_under_both_schedules(rt, cfg_id, flags):
    """The fused round (copies of the unconditioned rows, packing of the
    conditioned ones inside the finaliser) gives the same bits whichever
    schedule verifies."""
    f = {"default": 0, "raw": rt.COND_RAW, "overwrite": rt.COND_OVERWRITE,
         "none": rt.COND_NONE}[flags]
    x = make_round_inputs(CONFIGS[cfg_id], device="cuda")
    cfg = x["cfg"]
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = []
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        for mode in (rt.VERIFY_FULL, rt.VERIFY_WINDOWS, rt.VERIFY_WINDOWS):
            rt.retrace_set_verify_schedule(mode)
            outs.append(rt.run_round(x, ws, flags=f))
            torch.cuda.synchronize()
    finally:
        rt.retrace_set_verify_schedule(prev)
    for o in outs[1:]:
        for name in ("accept_len", "committed", "bonus", "n", "e_out"):
            assert torch.equal(getattr(o, name), getattr(outs[0], name)), name
    assert ws.check() == 0


@pytest.mark.parametrize("flags", ["default", "overwrite"])
def test_round_unaligned_e_out_both_schedules(rt, flags):
    """e_out one element off a 16-byte boundary: the copies after the windowed
    passes take their element-wise path; the bits equal the one-pass round's."""
    f = {"default": 0, "overwrite": rt.COND_OVERWRITE}[flags]
    x = make_round_inputs(CONFIGS[4], device="cuda")
    cfg = x["cfg"]
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = []
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        for mode in (rt.VERIFY_FULL, rt.VERIFY_WINDOWS):
            rt.retrace_set_verify_schedule(mode)
            out = rt.RoundBuffers(cfg.B, cfg.K, cfg.d, cfg.torch_dtype)
            big = torch.empty(cfg.B * cfg.K * cfg.d + 1, dtype=cfg.torch_dtype, device="cuda")
            out.e_out = big[1:].view(cfg.B, cfg.K, cfg.d)
            outs.append(rt.run_round(x, ws, out=out, flags=f))
            torch.cuda.synchronize()
    finally:
        rt.retrace_set_verify_schedule(prev)
    for name in ("accept_len", "committed", "bonus", "n", "e_out"):
        assert torch.equal(getattr(outs[1], name), getattr(outs[0], name)), name
    assert ws.check() == 0


# More sequences than the GB300's 152 SMs at a size the automatic schedule
# verifies in one pass: there the finalisers pack their own rows.
MANY_SEQUENCES = CONFIGS[2].__class__("bf16 B160 K8 d256 (one pass, copies in the finalisers)",
                                      160, 8, 4099, 256, "bf16", 1.0, "uniform", seed_offset=21)


@pytest.mark.parametrize("flags", ["default", "overwrite"])
def test_round_copies_in_finalisers_equal_copy_kernel(rt, flags):
    """One pass with at least as many sequences as SMs copies and packs rows
    inside the finalisers; the windowed schedule leaves them to the copy
    kernel.  Both give the same bits."""
    f = {"default": 0, "overwrite": rt.COND_OVERWRITE}[flags]
    x = make_round_inputs(MANY_SEQUENCES, device="cuda")
    cfg = x["cfg"]
    assert cfg.B >= torch.cuda.get_device_properties(0).multi_processor_count
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = []
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        for mode in (rt.VERIFY_FULL, rt.VERIFY_WINDOWS, rt.VERIFY_FULL):
            rt.retrace_set_verify_schedule(mode)
            outs.append(rt.run_round(x, ws, flags=f))
            torch.cuda.synchronize()
    finally:
        rt.retrace_set_verify_schedule(prev)
    want = oracle.verify(host_f64(x["logits"]), host_int(x["draft"]))
    np.testing.assert_array_equal(host_int(outs[0].accept_len), want["accept_len"])
    for o in outs[1:]:
        for name in ("accept_len", "committed", "bonus", "n", "e_out"):
            assert torch.equal(getattr(o, name), getattr(outs[0], name)), name
    assert ws.check() == 0
