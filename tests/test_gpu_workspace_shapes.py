"""One workspace, calls of changing shapes: results equal those of fresh workspaces.

The regions of a workspace that must be zero between calls (argmax keys,
tickets, counters) lie at offsets that depend on B and K, between regions
that hold data (live lists, packed-row offsets, the round's counters).  A
serving loop sizes one workspace for its largest batch and calls it with
whatever batch it has; every call must still see its counters at zero.
"""

import pytest
import torch

from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, make_sampled_inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def random_verify_case(B, K, V, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    logits = torch.randn((B, K + 1, V), generator=g, device="cuda").to(torch.bfloat16)
    draft = torch.argmax(logits[:, :K].float(), dim=-1).to(torch.int32)
    cut = torch.randint(0, K + 1, (B,), generator=g, device="cuda")
    draft = torch.where(torch.arange(K, device="cuda")[None, :] == cut[:, None], (draft + 1) % V, draft)
    return logits, draft


def verify(rt, logits, draft, ws):
    B, K1, _ = logits.shape
    outs = [torch.full((B,), -7, dtype=torch.int32, device="cuda"),
            torch.full((B, K1), -7, dtype=torch.int32, device="cuda"),
            torch.full((B,), -7, dtype=torch.int32, device="cuda")]
    rt.retrace_verify(logits, draft, *outs, ws)
    return outs


def test_changing_shapes_on_one_workspace(rt):
    big = CONFIGS[5]
    ws = rt.Workspace(big.B, big.K, big.V, big.d, big.torch_dtype)
    calls = []
    for cid in (4, 3, 5, 1):  # rounds of four shapes (d 2560, 4096, 256; bf16 and f32)
        cfg = CONFIGS[cid]
        x = make_round_inputs(cfg, device="cuda")
        calls.append(("round", cfg, x, None))
    x4 = make_round_inputs(CONFIGS[4], device="cuda")
    s4 = make_sampled_inputs(CONFIGS[4], x4["logits"], device="cuda")
    calls.insert(2, ("sampled", CONFIGS[4], x4, s4))
    for B, seed in ((128, 1), (32, 2), (200, 3)):  # greedy verification, windowed and one pass
        logits, draft = random_verify_case(B, 16, 151936, seed)
        calls.insert(1 + seed, ("verify", None, logits, draft))

    def run(kind, cfg, a, b, w):
        if kind == "round":
            out = rt.run_round(a, w)
            return [out.accept_len, out.committed, out.bonus, out.n, out.e_out]
        if kind == "sampled":
            out = rt.run_round_sampled(a, b, w)
            return [out.accept_len, out.committed, out.bonus, out.n, out.e_out]
        return verify(rt, a, b, w)

    for _ in range(2):  # twice over: every shape follows another
        for kind, cfg, a, b in calls:
            got = run(kind, cfg, a, b, ws)
            if kind == "verify":
                B, K1, V = a.shape
                fresh = rt.Workspace(B, K1 - 1, V, 8, a.dtype)
            else:
                fresh = rt.Workspace(cfg.B, cfg.K, cfg.V, cfg.d, cfg.torch_dtype)
            want = run(kind, cfg, a, b, fresh)
            torch.cuda.synchronize()
            for g, w in zip(got, want):
                assert torch.equal(g, w), kind
    assert ws.check() == 0
