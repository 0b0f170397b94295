"""GPU parity of the low-rank conditioning path (retrace_round_lowrank) vs the oracle.

Configs 1 (fp32, FFMA kernel), 3 and 4 (bf16, tensor cores) are checked in
full; a bf16 shape with d not a multiple of 128 takes the FFMA kernel; the
serving batch (config 5) is checked on its verification outputs, every
unconditioned row, and the conditioned rows of a seeded sample of sequences.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import assert_close, assert_verify_exact, host_f64, host_int
from paper_2608_29748_gb300.workloads import CONFIGS, make_lowrank_weights, make_round_inputs

pytestmark = pytest.mark.gpu

SIMT_BF16 = CONFIGS[2].__class__("bf16 d=320 (FFMA path)", 6, 16, 5003, 320, "bf16", 1.0, "uniform", seed_offset=9)


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def run(rt, x, w, ws=None, **kw):
    cfg = x["cfg"]
    if ws is None:
        ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    targ = torch.empty((cfg.B, cfg.K + 1), dtype=torch.int32, device="cuda")
    out = rt.run_round_lowrank(x, w, ws, target_argmax=targ, **kw)
    torch.cuda.synchronize()
    return out, targ, ws


def oracle_lowrank(x, w, seqs=None):
    dtype = "bf16" if x["logits"].dtype == torch.bfloat16 else "f32"
    sel = slice(None) if seqs is None else list(seqs)
    return oracle.retrace_round_lowrank(
        host_f64(x["logits"][sel]), host_int(x["draft"][sel]), host_f64(x["hD"][sel]), host_f64(x["hT"][sel]),
        host_f64(x["e"]), host_f64(w["P"]), host_f64(w["Bc"]), host_f64(w["Ac"]), host_f64(w["Wv_lr"]),
        host_f64(w["Wg_lr"]), x["beta"], dtype)


@pytest.mark.parametrize("cfg_id", [1, 3, 4, "simt-bf16"])
def test_lowrank_round_full(rt, cfg_id):
    cfg = SIMT_BF16 if cfg_id == "simt-bf16" else CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    w = make_lowrank_weights(cfg, device="cuda")
    out, targ, ws = run(rt, x, w)
    assert ws.check() == 0
    want = oracle_lowrank(x, w)
    assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
    np.testing.assert_array_equal(host_int(out.n), want["n"])
    assert_close(out.e_out, want["e_tilde"], f"config {cfg_id} low-rank e~")
    got, e = host_f64(out.e_out), host_f64(x["e"])
    for b in range(cfg.B):  # rows without a signal keep the mask embedding bit for bit
        assert np.array_equal(got[b, want["n"][b]:], np.broadcast_to(e, got[b, want["n"][b]:].shape))


def test_lowrank_serving_batch_sampled(rt):
    """Config 5 at full size (B=256, K=16, V=151936, d=4096) in the launch
    configuration the benchmark times."""
    cfg = CONFIGS[5]
    x = make_round_inputs(cfg, device="cuda")
    w = make_lowrank_weights(cfg, device="cuda")
    out, targ, ws = run(rt, x, w)
    assert ws.check() == 0
    ver = oracle.verify(host_f64(x["logits"]), host_int(x["draft"]))
    assert_verify_exact(ver, out.accept_len, out.committed, out.bonus, targ)
    n = oracle.carried_rows(ver["accept_len"], cfg.K)
    np.testing.assert_array_equal(host_int(out.n), n)
    pos = torch.arange(cfg.K, device="cuda")[None, :]
    mask = pos >= out.n.long()[:, None]
    assert torch.equal(out.e_out[mask], x["e"].expand(int(mask.sum()), cfg.d))
    rng = np.random.default_rng(7)
    carried = np.flatnonzero(n > 0)
    seqs = sorted({int(carried[0]), int(carried[-1]), *rng.choice(carried, size=6, replace=False).tolist()})
    want = oracle_lowrank(x, w, seqs)
    for i, b in enumerate(seqs):
        nb = int(n[b])
        assert_close(out.e_out[b, :nb], want["e_tilde"][i, :nb], f"config 5 sequence {b}")


def test_lowrank_short_blocks(rt):
    for K in (1, 2, 3):
        cfg = CONFIGS[2].__class__("t", 7, K, 4099, 256, "bf16", 1.0, "uniform", seed_offset=13)
        x = make_round_inputs(cfg, device="cuda")
        w = make_lowrank_weights(cfg, device="cuda")
        out, targ, ws = run(rt, x, w)
        want = oracle_lowrank(x, w)
        assert_verify_exact(want, out.accept_len, out.committed, out.bonus, targ)
        assert_close(out.e_out, want["e_tilde"], f"K={K}")
        if K == 1:
            assert torch.equal(out.e_out, x["e"].expand_as(out.e_out))


def test_lowrank_repeatable_bitwise_and_graph(rt):
    """The split partials are summed in a fixed order: repeated rounds on one
    workspace give identical bits, also when replayed from a CUDA graph."""
    x = make_round_inputs(CONFIGS[4], device="cuda")
    w = make_lowrank_weights(CONFIGS[4], device="cuda")
    first, _, ws = run(rt, x, w)
    for _ in range(3):
        again, _, _ = run(rt, x, w, ws=ws)
        assert torch.equal(again.e_out, first.e_out)
    out = rt.RoundBuffers(64, 16, 2560, torch.bfloat16)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        rt.run_round_lowrank(x, w, ws, out=out, stream=s)
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        rt.run_round_lowrank(x, w, ws, out=out, stream=s)
    out.e_out.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out.e_out, first.e_out)
    assert ws.check() == 0
