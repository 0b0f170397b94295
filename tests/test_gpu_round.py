"""GPU parity of the fused round (retrace_round) on the five workloads vs the oracle.

Configs 1-4 are checked in full.  Config 5 (B = 256, 1.3 GB of logits) is
checked twice: in full in the launch configuration the benchmark times
(target_argmax not requested, so the default schedule verifies in row
windows, copies and packs rows in the copy kernel and runs both projections
in cond_pair_kernel), and with target_argmax requested (one verification
pass) on a seeded sample of conditioned rows.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import assert_close, assert_verify_exact, host_f64, host_int, oracle_round
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def small_r_path(B, K, d):
    """Whether the conditioning of a bf16 round with a broadcast e takes the
    small-R GEMMs: at most 1024 possible rows, and the gate GEMM's work tiles
    (2d/128 weight tiles x N tiles of 256 rows) at most 256."""
    rows = (B * (K - 1) + 15) // 16 * 16
    return 0 < rows <= 1024 and (2 * d // 128) * ((rows + 255) // 256) <= 256


def run(rt, x, ws=None, **kw):
    cfg = x["cfg"]
    if ws is None:
        ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    targ = torch.empty((cfg.B, cfg.K + 1), dtype=torch.int32, device="cuda")
    out = rt.run_round(x, ws, target_argmax=targ, **kw)
    torch.cuda.synchronize()
    return out, targ, ws


@pytest.mark.parametrize("cfg_id", [1, 2, 3, 4])
def test_round_workloads_full(rt, cfg_id):
    x = make_round_inputs(CONFIGS[cfg_id], device="cuda")
    out, targ, ws = run(rt, x)
    assert ws.check() == 0
    want = oracle_round(x)
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
    np.testing.assert_array_equal(host_int(out.n), want["n"])
    assert_close(out.e_out, want["e_tilde"], f"config {cfg_id} e_tilde")
    # rows without an aligned signal keep the mask embedding bit-for-bit
    got = host_f64(out.e_out)
    e = host_f64(x["e"])
    for b in range(x["cfg"].B):
        assert np.array_equal(got[b, want["n"][b]:], np.broadcast_to(e, got[b, want["n"][b]:].shape))


def test_round_serving_batch_benched_path(rt):
    """Config 5 at full size (B=256, K=16, V=151936, d=4096) through exactly
    the call bench.py times: retrace_round with target_argmax NULL under the
    default schedule.  That composition is the row-window verification passes,
    verify_copy_kernel (unconditioned rows of e~, packing of [m; u]) and
    cond_pair_kernel (both projections; R = 2876 rows, so the last 256-row
    pair block is partial).  Every output is compared with the oracle: the
    verification outputs and n bit-exact, every row of e~ within the bf16
    tolerance, and the unconditioned rows bit-exact copies of e."""
    cfg = CONFIGS[5]
    windows = rt.retrace_verify_plan(cfg.B, cfg.K, cfg.V, cfg.torch_dtype)
    assert len(windows) > 2, "the default schedule verifies this workload in row windows"
    x = make_round_inputs(cfg, device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    out = rt.run_round(x, ws)  # no target_argmax: the benchmark's call
    torch.cuda.synchronize()
    assert ws.check() == 0
    want = oracle_round(x)
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus)
    np.testing.assert_array_equal(host_int(out.n), want["n"])
    R = int(want["n"].sum())
    assert R % 256 != 0 and R > 256, R  # several pair blocks and a partial last one
    assert_close(out.e_out, want["e_tilde"], "config 5 benched round, every row")
    pos = torch.arange(cfg.K, device="cuda")[None, :]
    mask = pos >= out.n.long()[:, None]
    assert torch.equal(out.e_out[mask], x["e"].expand(int(mask.sum()), cfg.d))


def test_round_serving_batch_sampled(rt):
    """Config 5 at full size with target_argmax requested (which makes the
    verification a single pass over every row): verification outputs in full,
    the unconditioned rows in full, a seeded sample of conditioned rows."""
    cfg = CONFIGS[5]
    x = make_round_inputs(cfg, device="cuda")
    out, targ, ws = run(rt, x)
    assert ws.check() == 0
    want = oracle.verify(host_f64(x["logits"]), host_int(x["draft"]))
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
    A = want["accept_len"]
    n = oracle.carried_rows(A, cfg.K)
    np.testing.assert_array_equal(host_int(out.n), n)
    # unconditioned rows: exact copies of e (checked on the device, all of them)
    pos = torch.arange(cfg.K, device="cuda")[None, :]
    mask = pos >= out.n.long()[:, None]
    assert torch.equal(out.e_out[mask], x["e"].expand(int(mask.sum()), cfg.d))
    # conditioned rows: a seeded sample, including the first and last rows of the plan
    rng = np.random.default_rng(42)
    cond = [(b, j) for b in range(cfg.B) for j in range(int(n[b]))]
    pick = sorted({0, len(cond) - 1, *rng.choice(len(cond), size=40, replace=False).tolist()})
    rows = [cond[i] for i in pick]
    ref = oracle.conditioned_rows(rows, A, host_f64(x["hD"]), host_f64(x["hT"]), host_f64(x["e"]),
                                  host_f64(x["Wc"]), host_f64(x["Wv"]), host_f64(x["Wg"]), x["beta"], "bf16")
    got = torch.stack([out.e_out[b, j] for b, j in rows])
    assert_close(got, ref, "config 5 sampled rows")


def test_round_dense_e_and_short_blocks(rt):
    """Per-position e ([B, K, d]) and blocks of 1 and 2 drafts."""
    for K in (1, 2, 16):
        cfg = CONFIGS[2].__class__("t", 9, K, 3001, 512, "bf16", 1.0, "uniform", seed_offset=7)
        x = make_round_inputs(cfg, device="cuda")
        x["e"] = (torch.randn((cfg.B, K, cfg.d), device="cuda") * 0.02).to(torch.bfloat16)
        out, targ, ws = run(rt, x)
        want = oracle_round(x)
        assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
        assert_close(out.e_out, want["e_tilde"], f"K={K}")
        if K == 1:  # a one-token block never carries anything: e~ == e
            assert torch.equal(out.e_out, x["e"])


def test_round_in_cuda_graph(rt):
    """The round captures into a CUDA graph (no host sync, no allocation) and replays exactly."""
    x = make_round_inputs(CONFIGS[4], device="cuda")
    eager, targ, ws = run(rt, x)
    out = rt.RoundBuffers(64, 16, 2560, torch.bfloat16)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        rt.run_round(x, ws, out=out, stream=s)  # warm-up on the capture stream
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        rt.run_round(x, ws, out=out, stream=s)
    for _ in range(3):
        out.e_out.zero_()
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out.e_out, eager.e_out)
    assert torch.equal(out.committed, eager.committed)
    assert ws.check() == 0


def test_round_phase_events(rt):
    x = make_round_inputs(CONFIGS[3], device="cuda")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    for e in ev:
        e.record()  # creates the underlying CUDA events
    run(rt, x, phase_events=ev)
    t = [ev[i].elapsed_time(ev[i + 1]) for i in range(3)]
    assert all(v >= 0 for v in t)


def test_round_repeatable_bitwise(rt):
    """Packed rows are claimed with atomics, so their order varies from run to
    run; every output row depends only on its own inputs, so the results must
    not: five rounds on one workspace give identical bits."""
    x = make_round_inputs(CONFIGS[4], device="cuda")
    first, targ, ws = run(rt, x)
    for _ in range(4):
        again, _, _ = run(rt, x, ws=ws)
        assert torch.equal(again.e_out, first.e_out)
        assert torch.equal(again.committed, first.committed)
        assert torch.equal(again.accept_len, first.accept_len)
    assert ws.check() == 0


@pytest.mark.parametrize("cfg_id", [3, 4])
def test_overlapped_round_equals_separate_entry_points(rt, cfg_id):
    """retrace_round with RETRACE_ROUND_OVERLAP (verification and both
    projections overlapped in one persistent kernel) against retrace_verify +
    retrace_align_refine + retrace_gate_fuse on the same inputs: identical
    bits, since every output element is computed by the same arithmetic in
    the same order -- except where the separate entry points take the
    small-R path (split-K sums, another fp32 summation order), where both
    must match the oracle instead."""
    x = make_round_inputs(CONFIGS[cfg_id], device="cuda")
    cfg = x["cfg"]
    fused, targ, ws = run(rt, x, flags=rt.ROUND_OVERLAP)
    B, K, d = cfg.B, cfg.K, cfg.d
    acc = torch.empty(B, dtype=torch.int32, device="cuda")
    com = torch.empty(B, K + 1, dtype=torch.int32, device="cuda")
    bon = torch.empty(B, dtype=torch.int32, device="cuda")
    r = torch.empty(B, K, d, dtype=torch.bfloat16, device="cuda")
    n = torch.empty(B, dtype=torch.int32, device="cuda")
    e_out = torch.empty(B, K, d, dtype=torch.bfloat16, device="cuda")
    rt.retrace_verify(x["logits"], x["draft"], acc, com, bon, ws)
    rt.retrace_align_refine(x["hD"], x["hT"], acc, x["Wc"], x["beta"], r, n, ws)
    rt.retrace_gate_fuse(x["e"], r, n, x["Wv"], x["Wg"], e_out, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    assert torch.equal(acc, fused.accept_len)
    assert torch.equal(com, fused.committed)
    assert torch.equal(bon, fused.bonus)
    assert torch.equal(n, fused.n)
    if small_r_path(B, K, d):
        want = oracle_round(x)
        assert_close(fused.e_out, want["e_tilde"], "overlapped round")
        assert_close(e_out, want["e_tilde"], "separate entry points, small-R path")
    else:
        assert torch.equal(e_out, fused.e_out)


def test_overlapped_round_matches_the_oracle_and_the_default_path(rt):
    """The overlapped kernel on the serving shape's sibling (B = 64): oracle
    parity, and the default round's outputs (the same bits where both take
    the same GEMMs; at B = 64 the default round takes the small-R path, so
    both are held to the oracle)."""
    x = make_round_inputs(CONFIGS[4], device="cuda")
    over, targ, ws = run(rt, x, flags=rt.ROUND_OVERLAP)
    assert ws.check() == 0
    want = oracle_round(x)
    assert_verify_exact(want, over.accept_len, over.committed, over.bonus, targ)
    assert_close(over.e_out, want["e_tilde"], "overlapped round")
    plain, _, _ = run(rt, x, ws=ws)
    assert torch.equal(plain.n, over.n)
    cfg = x["cfg"]
    if small_r_path(cfg.B, cfg.K, cfg.d):
        assert_close(plain.e_out, want["e_tilde"], "default round, small-R path")
    else:
        assert torch.equal(plain.e_out, over.e_out)


def test_overlap_flag_rejects_what_the_kernel_does_not_cover(rt):
    """RETRACE_ROUND_OVERLAP on an fp32 round or with an ablation flag is
    refused with UNSUPPORTED before anything is enqueued."""
    x = make_round_inputs(CONFIGS[1], device="cuda")  # fp32
    with pytest.raises(rt.RetraceError) as ei:
        run(rt, x, flags=rt.ROUND_OVERLAP)
    assert ei.value.status == 2
    x = make_round_inputs(CONFIGS[3], device="cuda")
    with pytest.raises(rt.RetraceError) as ei:
        run(rt, x, flags=rt.ROUND_OVERLAP | rt.COND_RAW)
    assert ei.value.status == 2


# Ablation variants (component ablation, Table 3): raw conditioning gated,
# raw conditioning overwrite, no conditioning.
SMALL_SIMT_BF16 = CONFIGS[2].__class__("bf16 d=320 (FFMA path)", 6, 16, 5003, 320, "bf16", 1.0, "uniform", seed_offset=9)


def _flag(rt, variant):
    return {"raw": rt.COND_RAW, "overwrite": rt.COND_OVERWRITE, "none": rt.COND_NONE}[variant]


@pytest.mark.parametrize("variant", ["raw", "overwrite", "none"])
@pytest.mark.parametrize("cfg_id", [1, 3, 4, "simt-bf16"])
def test_ablation_variants(rt, cfg_id, variant):
    cfg = SMALL_SIMT_BF16 if cfg_id == "simt-bf16" else CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    if variant != "raw":  # weights the variant does not use may be absent
        x = {**x, "Wc": None, "Wv": None, "Wg": None}
    else:
        x = {**x, "Wc": None}
    out, targ, ws = run(rt, x, flags=_flag(rt, variant))
    assert ws.check() == 0
    want = oracle_round(x, variant)
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
    np.testing.assert_array_equal(host_int(out.n), want["n"])
    if variant == "raw":
        assert_close(out.e_out, want["e_tilde"], f"config {cfg_id} raw")
    else:  # pure copies: bit-exact
        assert np.array_equal(host_f64(out.e_out), want["e_tilde"]), f"config {cfg_id} {variant}"


@pytest.mark.parametrize("variant", ["raw", "overwrite", "none"])
def test_ablation_variants_dense_e_and_short_blocks(rt, variant):
    for K in (1, 2, 16):
        cfg = CONFIGS[2].__class__("t", 9, K, 3001, 512, "bf16", 1.0, "uniform", seed_offset=11)
        x = make_round_inputs(cfg, device="cuda")
        x["e"] = (torch.randn((cfg.B, K, cfg.d), device="cuda") * 0.02).to(torch.bfloat16)
        out, targ, ws = run(rt, x, flags=_flag(rt, variant))
        want = oracle_round(x, variant)
        assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
        if variant == "raw":
            assert_close(out.e_out, want["e_tilde"], f"K={K} raw")
        else:
            assert np.array_equal(host_f64(out.e_out), want["e_tilde"]), f"K={K} {variant}"


def test_raw_variant_equals_zero_beta_on_the_default_path(rt):
    """Raw conditioning skips the correction GEMM; beta = 0 runs it and adds
    0 * c: both give r = m, so the outputs agree bit for bit."""
    x = make_round_inputs(CONFIGS[4], device="cuda")
    raw, _, ws = run(rt, x, flags=rt.COND_RAW)
    zero, _, _ = run(rt, {**x, "beta": 0.0}, ws=ws)
    assert torch.equal(raw.e_out, zero.e_out)


@pytest.mark.parametrize("R", [0, 1])
def test_small_r_round_with_almost_nothing_to_condition(rt, R):
    """Config 3's shapes (small-R GEMMs) with every draft accepted (R = 0: no
    row is conditioned, the GEMMs' CTAs all idle) or all but one row (R = 1):
    e~ keeps e bit for bit wherever no signal is carried, and the one
    conditioned row matches the oracle."""
    cfg = CONFIGS[3]
    x = make_round_inputs(cfg, device="cuda")
    top = torch.argmax(x["logits"][:, : cfg.K].float(), dim=-1).to(torch.int32)
    x["draft"] = top.clone()
    if R == 1:  # sequence 0 rejects its draft at position K-2: n_0 = 1
        x["draft"][0, cfg.K - 2] = (top[0, cfg.K - 2] + 1) % cfg.V
    out, targ, ws = run(rt, x)
    assert ws.check() == 0
    want = oracle_round(x)
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
    assert int(out.n.sum()) == R
    assert_close(out.e_out, want["e_tilde"], f"R={R}")
    got = host_f64(out.e_out)
    e = host_f64(x["e"])
    for b in range(cfg.B):
        nb = int(want["n"][b])
        assert np.array_equal(got[b, nb:], np.broadcast_to(e, got[b, nb:].shape))
