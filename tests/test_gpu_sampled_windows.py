"""Windowed schedule of stochastic verification vs the one-pass schedule and the oracle.

The outputs of speculative sampling depend only on the target rows 0..A_b and
the drafter rows 0..min(A_b, K-1): the accept tests stop at the first
rejection, whose row also gives the residual draw.  The windowed schedule
scans the row windows of the sequences that accepted every earlier draft, and
its outputs must equal the one-pass schedule's bit for bit (both decide from
the same per-row top-k lists) and the oracle's.  Acceptance is planted here
so that every window boundary is crossed: drafter rows equal to the target's
(q = p, so a draft in the kept set is always accepted) and, at row a_b, a
draft outside the target's top k (p = 0: always rejected).
"""

import numpy as np
import pytest
import torch

from parity import host_int
from test_gpu_sampled import check_against_oracle
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, make_sampled_inputs

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


def sampled(rt, x, s, ws, T, k, p):
    B, K1, _ = x["logits"].shape
    outs = [torch.full((B,), -7, dtype=torch.int32, device="cuda"),
            torch.full((B, K1), -7, dtype=torch.int32, device="cuda"),
            torch.full((B,), -7, dtype=torch.int32, device="cuda")]
    rt.retrace_verify_sampled(x["logits"], s["draft_logits"], s["draft"], s["uniforms"], T, k, p, *outs, ws)
    torch.cuda.synchronize()
    return outs


def planted(cfg, accept):
    """Target logits of cfg; drafter rows = target rows; drafts = the target's
    argmax in rows i < a_b and its smallest logit's index in row a_b."""
    x = make_round_inputs(cfg, device="cuda")
    tl = x["logits"]
    B, K1, V = tl.shape
    K = K1 - 1
    s = make_sampled_inputs(cfg, tl, device="cuda")
    s["draft_logits"] = tl[:, :K].contiguous()
    top = torch.argmax(tl[:, :K].float(), dim=-1)
    low = torch.argmin(tl[:, :K].float(), dim=-1)
    i = torch.arange(K, device="cuda")[None, :]
    a = accept.to("cuda")[:, None]
    s["draft"] = torch.where(i < a, top, low).to(torch.int32)
    return x, s


@pytest.mark.parametrize("cfg_id", [1, 3, 4])
@pytest.mark.parametrize("T,k,p", [(1.0, 20, 0.95), (0.7, 64, 0.8), (1.3, 5, 1.0)])
def test_windowed_equals_one_pass(rt, cfg_id, T, k, p):
    cfg = CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        full = sampled(rt, x, s, ws, T, k, p)
        rt.retrace_set_verify_schedule(rt.VERIFY_WINDOWS)
        for _ in range(2):  # and again on the same workspace
            win = sampled(rt, x, s, ws, T, k, p)
            for a, b in zip(win, full):
                assert torch.equal(a, b)
    finally:
        rt.retrace_set_verify_schedule(prev)
    assert ws.check() == 0


@pytest.mark.parametrize("cfg_id", [3, 4])
def test_windowed_planted_acceptance_every_boundary(rt, windows, cfg_id):
    cfg = CONFIGS[cfg_id]
    accept = torch.arange(cfg.B) % (cfg.K + 1)  # every accepted length 0..K
    x, s = planted(cfg, accept)
    acc = check_against_oracle(rt, x, s)
    np.testing.assert_array_equal(acc, accept.numpy())


def test_windowed_all_accepted(rt, windows):
    cfg = CONFIGS[4]
    x, s = planted(cfg, torch.full((cfg.B,), cfg.K))
    acc = check_against_oracle(rt, x, s)
    assert (acc == cfg.K).all()


@pytest.mark.parametrize("cfg_id", [1, 3, 4])
def test_windowed_round_equals_one_pass(rt, cfg_id):
    """The round: outputs, n and e~ (copies and packing after the last pass,
    then the projections) equal the one-pass round's bit for bit."""
    cfg = CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = []
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        for mode in (rt.VERIFY_FULL, rt.VERIFY_WINDOWS):
            rt.retrace_set_verify_schedule(mode)
            outs.append(rt.run_round_sampled(x, s, ws))
            torch.cuda.synchronize()
    finally:
        rt.retrace_set_verify_schedule(prev)
    for name in ("accept_len", "committed", "bonus", "n", "e_out"):
        assert torch.equal(getattr(outs[1], name), getattr(outs[0], name)), name
    assert host_int(outs[1].n).sum() > 0
    assert ws.check() == 0


@pytest.mark.parametrize("K", [5, 6, 9, 11])
def test_windowed_short_blocks(rt, K):
    """Windows [0,4),[4,6) at K = 5 (the last window has one target row, K,
    and one drafter row, 4), [0,4),[4,7) at K = 6, [0,4),[4,10) at K = 9 and
    [0,4),[4,12) at K = 11: equal to the one-pass schedule, accepted lengths
    from 0 to K planted."""
    cfg = CONFIGS[2].__class__(f"sampled-K{K}", K + 1, K, 3001, 8, "bf16", 1.0, "uniform", seed_offset=40 + K)
    accept = torch.arange(cfg.B) % (K + 1)
    x, s = planted(cfg, accept)
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        full = sampled(rt, x, s, ws, 1.0, 20, 0.95)
        rt.retrace_set_verify_schedule(rt.VERIFY_WINDOWS)
        assert len(rt.retrace_verify_plan(cfg.B, K, cfg.V, cfg.torch_dtype)) == 3
        win = sampled(rt, x, s, ws, 1.0, 20, 0.95)
    finally:
        rt.retrace_set_verify_schedule(prev)
    for a, b in zip(win, full):
        assert torch.equal(a, b)
    np.testing.assert_array_equal(host_int(win[0]), accept.numpy())
    assert ws.check() == 0


def test_one_pass_round_many_sequences_equals_windowed(rt):
    """More sequences than the GB300's 152 SMs: the one-pass round's finalisers
    copy and pack their own rows, the windowed round leaves them to the copy
    kernel.  Both give the same bits."""
    cfg = CONFIGS[2].__class__("sampled bf16 B160 K8 d256", 160, 8, 4096, 256, "bf16", 1.0, "uniform",
                               seed_offset=23)
    assert cfg.B >= torch.cuda.get_device_properties(0).multi_processor_count
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = []
    prev = rt.retrace_set_verify_schedule(rt.VERIFY_FULL)
    try:
        for mode in (rt.VERIFY_FULL, rt.VERIFY_WINDOWS, rt.VERIFY_FULL):
            rt.retrace_set_verify_schedule(mode)
            outs.append(rt.run_round_sampled(x, s, ws))
            torch.cuda.synchronize()
    finally:
        rt.retrace_set_verify_schedule(prev)
    for o in outs[1:]:
        for name in ("accept_len", "committed", "bonus", "n", "e_out"):
            assert torch.equal(getattr(o, name), getattr(outs[0], name)), name
    assert ws.check() == 0


def test_greedy_and_sampled_windows_share_a_workspace(rt, windows):
    """Windowed greedy and windowed temperature-T verification alternate on
    one workspace: each must leave the live lists, pass counters and keys as
    the other expects, so every call equals the same call on a fresh
    workspace (and the greedy one equals the oracle)."""
    import oracle
    from parity import host_f64

    cfg = CONFIGS[4]
    g = torch.Generator()
    g.manual_seed(123)
    accept = torch.randint(0, cfg.K + 1, (cfg.B,), generator=g)
    x, s = planted(cfg, accept)
    T, k, p = s["temperature"], s["top_k"], s["top_p"]

    def greedy(ws):
        B, K1, _ = x["logits"].shape
        outs = [torch.full((B,), -7, dtype=torch.int32, device="cuda"),
                torch.full((B, K1), -7, dtype=torch.int32, device="cuda"),
                torch.full((B,), -7, dtype=torch.int32, device="cuda")]
        rt.retrace_verify(x["logits"], s["draft"], *outs, ws)
        torch.cuda.synchronize()
        return outs

    def fresh():
        return rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)

    ref_g, ref_s = greedy(fresh()), sampled(rt, x, s, fresh(), T, k, p)
    want = oracle.verify(host_f64(x["logits"]), host_int(s["draft"]))
    np.testing.assert_array_equal(host_int(ref_g[0]), want["accept_len"])
    np.testing.assert_array_equal(host_int(ref_g[1]), want["committed"])
    ws = fresh()
    for it in range(6):
        got, ref = (greedy(ws), ref_g) if it % 2 == 0 else (sampled(rt, x, s, ws, T, k, p), ref_s)
        for a, b in zip(got, ref):
            assert torch.equal(a, b), it
    assert ws.check() == 0
