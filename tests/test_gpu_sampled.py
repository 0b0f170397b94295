"""GPU parity of stochastic verification (retrace_verify_sampled) vs the oracle.

Floating point decides the accept tests, the top-p cut and the draws; the GPU
computes them in fp32 and the oracle in float64.  The uniforms are inputs, so
the tests move any uniform that lies within a small margin of its decision
boundary (measure-zero cases) and mark the sequences whose top-p cut itself is
that close; those sequences are checked for validity instead of equality.
The lossless property is checked on the GPU's own draws.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import host_f64, host_int
from sampling import _dist, conditioned_uniforms
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, make_sampled_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def run(rt, tl, dl, draft, u, T, k, p, dtype):
    B, K1, V = tl.shape
    K = K1 - 1
    ws = rt.Workspace(B, K, V, 1, dtype)
    acc = torch.empty(B, dtype=torch.int32, device="cuda")
    com = torch.empty(B, K1, dtype=torch.int32, device="cuda")
    bon = torch.empty(B, dtype=torch.int32, device="cuda")
    rt.retrace_verify_sampled(tl, dl, draft, u, T, k, p, acc, com, bon, ws)
    torch.cuda.synchronize()
    assert ws.check() == 0
    return host_int(acc), host_int(com), host_int(bon)


def check_against_oracle(rt, x, s, T=None, k=None, p=None):
    T = s["temperature"] if T is None else T
    k = s["top_k"] if k is None else k
    p = s["top_p"] if p is None else p
    tl, dl = host_f64(x["logits"]), host_f64(s["draft_logits"])
    draft = host_int(s["draft"])
    u, amb = conditioned_uniforms(tl, dl, draft, s["uniforms"].cpu().numpy().astype(np.float64), T, k, p)
    u_dev = torch.tensor(u, dtype=torch.float32, device="cuda")
    acc, com, bon = run(rt, x["logits"], s["draft_logits"], s["draft"], u_dev, T, k, p, x["logits"].dtype)
    want = oracle.verify_sampled(tl, dl, draft, u_dev.cpu().double().numpy(), T, k, p)
    B = draft.shape[0]
    exact = [b for b in range(B) if b not in amb]
    assert len(exact) >= 0.9 * B
    np.testing.assert_array_equal(acc[exact], want["accept_len"][exact])
    np.testing.assert_array_equal(com[exact], want["committed"][exact])
    np.testing.assert_array_equal(bon[exact], want["bonus"][exact])
    for b in amb:  # valid, if not necessarily the oracle's choice at a boundary
        a = int(acc[b])
        assert (com[b, :a] == draft[b, :a]).all() and (com[b, a + 1:] == -1).all() and com[b, a] == bon[b]
        toks, _ = _dist(tl[b, a], T, k, 1.0)
        assert bon[b] in toks
    return acc


@pytest.mark.parametrize("cfg_id", [1, 3, 4])
def test_sampled_verification_matches_the_oracle(rt, cfg_id):
    cfg = CONFIGS[cfg_id]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    acc = check_against_oracle(rt, x, s)
    if cfg.B > 1:
        assert 0 < acc.mean() < cfg.K  # a realistic mix of accepted and rejected drafts


@pytest.mark.parametrize("T,k,p", [(1.0, 1, 0.95), (0.7, 64, 0.8), (1.3, 5, 1.0), (1.0, 20, 0.3)])
def test_sampled_verification_parameters(rt, T, k, p):
    cfg = CONFIGS[2].__class__("sampled", 12, 5, 3001, 8, "bf16", 1.0, "uniform", seed_offset=21)
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    check_against_oracle(rt, x, s, T, k, p)


def test_sampled_verification_with_top_k_one_is_greedy(rt):
    """top_k = 1 with drafts at the drafter's argmax: the greedy kernel's outputs, bit for bit."""
    cfg = CONFIGS[4]
    x = make_round_inputs(cfg, device="cuda")
    s = make_sampled_inputs(cfg, x["logits"], device="cuda")
    draft = torch.argmax(s["draft_logits"].float(), dim=-1).to(torch.int32)
    B, K = draft.shape
    ws = rt.Workspace(B, K, cfg.V, cfg.d, cfg.torch_dtype)
    outs = [torch.empty(B, dtype=torch.int32, device="cuda"), torch.empty(B, K + 1, dtype=torch.int32, device="cuda"),
            torch.empty(B, dtype=torch.int32, device="cuda")]
    rt.retrace_verify_sampled(x["logits"], s["draft_logits"], draft, s["uniforms"], 1.0, 1, 0.95, *outs, ws)
    greedy = [torch.empty_like(o) for o in outs]
    rt.retrace_verify(x["logits"], draft, *greedy, ws)
    torch.cuda.synchronize()
    for a, b in zip(outs, greedy):
        assert torch.equal(a, b)


def test_sampled_verification_is_lossless_on_the_gpu(rt):
    """Over many independent uniforms, the GPU's first committed token is
    distributed as the filtered target distribution p_0 (drafts drawn from q)."""
    B, K, V, T, k, p = 200_000, 2, 96, 1.0, 20, 0.95
    g = torch.Generator(device="cpu").manual_seed(5)
    tl1 = (torch.randn((K + 1, V), generator=g) * 1.5).to(torch.bfloat16)
    dl1 = (tl1[:K].float() + torch.randn((K, V), generator=g) * 0.8).to(torch.bfloat16)
    qt, qp = _dist(host_f64(dl1[0]), T, k, p)
    pick = torch.multinomial(torch.tensor(qp), B, replacement=True, generator=g)
    draft = torch.zeros((B, K), dtype=torch.int32)
    draft[:, 0] = torch.tensor(qt)[pick].to(torch.int32)
    draft[:, 1] = int(np.argmax(host_f64(dl1[1])))
    tl = tl1.expand(B, K + 1, V).contiguous().cuda()
    dl = dl1.expand(B, K, V).contiguous().cuda()
    u = torch.rand((B, K + 1), generator=g).cuda()
    acc, com, _ = run(rt, tl, dl, draft.cuda(), u, T, k, p, torch.bfloat16)
    pt, pp = _dist(host_f64(tl1[0]), T, k, p)
    freq = np.bincount(com[:, 0], minlength=V) / B
    want = np.zeros(V)
    want[pt] = pp
    sd = np.sqrt(np.maximum(want * (1 - want), 1e-12) / B)
    assert np.all(np.abs(freq - want) <= 5 * sd + 1e-4), np.max(np.abs(freq - want) / (sd + 1e-12))
