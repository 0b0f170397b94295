"""GPU parity of the temperature-T round (retrace_round_sampled) vs the oracle.

The verification part equals retrace_verify_sampled bit for bit (same
kernels) and the oracle's speculative sampling on every sequence whose
decisions are not within rounding of a boundary (helpers in sampling.py).
The conditioning part is a deterministic function of the accepted lengths:
it is checked against the oracle's Eq. 4-8 evaluated at the GPU's A_b.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import assert_close, host_f64, host_int
from sampling import conditioned_uniforms
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, make_sampled_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def conditioned_uniforms_for(x, s, seqs=None):
    sel = slice(None) if seqs is None else list(seqs)
    tl, dl = host_f64(x["logits"][sel]), host_f64(s["draft_logits"][sel])
    draft = host_int(s["draft"][sel])
    u, amb = conditioned_uniforms(tl, dl, draft, s["uniforms"][sel].cpu().numpy().astype(np.float64),
                                  s["temperature"], s["top_k"], s["top_p"])
    return tl, dl, draft, u, amb


def standalone_verify(rt, x, s, ws):
    B, K1, _ = x["logits"].shape
    outs = [torch.empty(B, dtype=torch.int32, device="cuda"), torch.empty(B, K1, dtype=torch.int32, device="cuda"),
            torch.empty(B, dtype=torch.int32, device="cuda")]
    rt.retrace_verify_sampled(x["logits"], s["draft_logits"], s["draft"], s["uniforms"], s["temperature"],
                              s["top_k"], s["top_p"], *outs, ws)
    return outs


def check_conditioning(x, out, rows, dtype):
    A = host_int(out.accept_len)
    ref = oracle.conditioned_rows(rows, A, host_f64(x["hD"]), host_f64(x["hT"]), host_f64(x["e"]),
                                  host_f64(x["Wc"]), host_f64(x["Wv"]), host_f64(x["Wg"]), x["beta"], dtype)
    got = torch.stack([out.e_out[b, j] for b, j in rows])
    assert_close(got, ref, "sampled round e~")


def check_round(rt, x, s):
    cfg_B, K1, _ = x["logits"].shape
    K = K1 - 1
    d = x["hD"].shape[2]
    dtype = "bf16" if x["logits"].dtype == torch.bfloat16 else "f32"
    tl, dl, draft, u, amb = conditioned_uniforms_for(x, s)
    s = dict(s, uniforms=torch.tensor(u, dtype=torch.float32, device="cuda"))
    ws = rt.Workspace(cfg_B, K, x["logits"].shape[2], d, x["logits"].dtype)
    out = rt.run_round_sampled(x, s, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    # verification: the standalone kernels' outputs, and the oracle's where unambiguous
    alone = standalone_verify(rt, x, s, ws)
    torch.cuda.synchronize()
    for a, b in zip((out.accept_len, out.committed, out.bonus), alone):
        assert torch.equal(a, b)
    want = oracle.verify_sampled(tl, dl, draft, u, s["temperature"], s["top_k"], s["top_p"])
    exact = [b for b in range(cfg_B) if b not in amb]
    np.testing.assert_array_equal(host_int(out.accept_len)[exact], want["accept_len"][exact])
    np.testing.assert_array_equal(host_int(out.committed)[exact], want["committed"][exact])
    A = host_int(out.accept_len)
    n = oracle.carried_rows(A, K)
    np.testing.assert_array_equal(host_int(out.n), n)
    # conditioning at the GPU's A_b (Eq. 4-8, batched): every row
    hD, hT = host_f64(x["hD"]), host_f64(x["hT"])
    m, uu = oracle.align(hD, hT, A)
    e_full = np.broadcast_to(host_f64(x["e"]), hD.shape)
    _, e_tilde = oracle.condition(e_full, m, uu, n, host_f64(x["Wc"]), host_f64(x["Wv"]), host_f64(x["Wg"]),
                                  x["beta"], "corrected", round_r_bf16=(dtype == "bf16"))
    assert_close(out.e_out, e_tilde, "sampled round e~")
    got = host_f64(out.e_out)
    for b in range(cfg_B):  # rows without a signal keep e bit for bit
        assert np.array_equal(got[b, n[b]:], np.broadcast_to(host_f64(x["e"]), hD.shape)[b, n[b]:])
    return out


@pytest.mark.parametrize("cfg_id", [1, 3, 4])
def test_sampled_round_matches_the_oracle(rt, cfg_id):
    cfg = CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    out = check_round(rt, x, s)
    if cfg.B > 1:
        assert 0 < host_int(out.n).sum()  # some sequences carry a rejected suffix


def test_sampled_round_dense_e_and_short_blocks(rt):
    """Per-position e (packed by the finalize kernel) and blocks of 1 and 2 drafts,
    on the tensor-core (d = 512) and FFMA (d = 320) conditioning paths."""
    for K, d in ((1, 512), (2, 512), (16, 512), (16, 320)):
        cfg = CONFIGS[2].__class__("t", 9, K, 3001, d, "bf16", 1.0, "uniform", seed_offset=17)
        x = make_round_inputs(cfg, device="cuda")
        x["e"] = (torch.randn((cfg.B, K, cfg.d), device="cuda") * 0.02).to(torch.bfloat16)
        s = make_sampled_inputs(cfg, x["logits"], device="cuda")
        out = check_round(rt, x, s)
        if K == 1:
            assert torch.equal(out.e_out, x["e"])


def test_sampled_round_serving_batch(rt):
    """Config 5 at full size (B=256, K=16, V=151936, d=4096) in the launch
    configuration the benchmark times: verification on a seeded sample of
    sequences against the oracle, every unconditioned row, and a sample of
    conditioned rows."""
    cfg = CONFIGS[5]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    out = rt.run_round_sampled(x, s, ws)
    alone = standalone_verify(rt, x, s, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    for a, b in zip((out.accept_len, out.committed, out.bonus), alone):
        assert torch.equal(a, b)
    rng = np.random.default_rng(11)
    seqs = sorted(rng.choice(cfg.B, size=8, replace=False).tolist())
    tl, dl, draft, u, amb = conditioned_uniforms_for(x, s, seqs)
    s2 = {k: (v[seqs].contiguous() if torch.is_tensor(v) else v) for k, v in s.items()}
    s2["uniforms"] = torch.tensor(u, dtype=torch.float32, device="cuda")
    x2 = {k: (v[seqs].contiguous() if torch.is_tensor(v) and v.dim() == 3 else v) for k, v in x.items()}
    sub = rt.run_round_sampled(x2, s2, rt.Workspace(len(seqs), cfg.K, cfg.V, cfg.d, cfg.torch_dtype))
    torch.cuda.synchronize()
    want = oracle.verify_sampled(tl, dl, draft, u, s["temperature"], s["top_k"], s["top_p"])
    exact = [i for i in range(len(seqs)) if i not in amb]
    np.testing.assert_array_equal(host_int(sub.accept_len)[exact], want["accept_len"][exact])
    np.testing.assert_array_equal(host_int(sub.committed)[exact], want["committed"][exact])
    n = oracle.carried_rows(host_int(out.accept_len), cfg.K)
    np.testing.assert_array_equal(host_int(out.n), n)
    assert 0 < n.sum()
    pos = torch.arange(cfg.K, device="cuda")[None, :]
    mask = pos >= out.n.long()[:, None]
    assert torch.equal(out.e_out[mask], x["e"].expand(int(mask.sum()), cfg.d))
    cond = [(b, j) for b in range(cfg.B) for j in range(int(n[b]))]
    pick = sorted({0, len(cond) - 1, *rng.choice(len(cond), size=40, replace=False).tolist()})
    check_conditioning(x, out, [cond[i] for i in pick], "bf16")


def test_sampled_round_in_cuda_graph(rt):
    """The sampled round captures into a CUDA graph and replays exactly."""
    cfg = CONFIGS[4]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    ws = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
    eager = rt.run_round_sampled(x, s, ws)
    torch.cuda.synchronize()
    out = rt.RoundBuffers(cfg.B, cfg.K, cfg.d, cfg.torch_dtype)
    st = torch.cuda.Stream()
    st.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(st):
        rt.run_round_sampled(x, s, ws, out=out, stream=st)
    torch.cuda.current_stream().wait_stream(st)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=st):
        rt.run_round_sampled(x, s, ws, out=out, stream=st)
    for _ in range(2):
        out.e_out.zero_()
        g.replay()
    torch.cuda.synchronize()
    assert ws.check() == 0
    for a, b in ((out.accept_len, eager.accept_len), (out.committed, eager.committed), (out.n, eager.n),
                 (out.e_out, eager.e_out)):
        assert torch.equal(a, b)
