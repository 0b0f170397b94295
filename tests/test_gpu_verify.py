"""GPU parity of greedy verification (argmax, first mismatch, commit) vs the oracle.

Every output is integer-valued and must match the oracle bit-exactly.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import assert_verify_exact, host_f64, host_int
from paper_2608_29748_gb300.workloads import CONFIGS, make_round_inputs, plant_prefix

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def rt():
    from paper_2608_29748_gb300 import binding

    return binding


def run_verify(rt, logits, draft, ws=None):
    B, K1, V = logits.shape
    K = K1 - 1
    dev = logits.device
    if ws is None:
        ws = rt.Workspace(B, K, V, 8, logits.dtype)
    acc = torch.full((B,), -7, dtype=torch.int32, device=dev)
    com = torch.full((B, K + 1), -7, dtype=torch.int32, device=dev)
    bon = torch.full((B,), -7, dtype=torch.int32, device=dev)
    targ = torch.full((B, K + 1), -7, dtype=torch.int32, device=dev)
    rt.retrace_verify(logits, draft, acc, com, bon, ws, target_argmax=targ)
    torch.cuda.synchronize()
    return acc, com, bon, targ


def check_against_oracle(rt, logits, draft, ws=None):
    acc, com, bon, targ = run_verify(rt, logits, draft, ws)
    want = oracle.verify(host_f64(logits), host_int(draft))
    assert_verify_exact(want, acc, com, bon, targ)
    return want


@pytest.mark.parametrize("cfg_id", [1, 2, 3, 4])
def test_verify_workloads(rt, cfg_id):
    x = make_round_inputs(CONFIGS[cfg_id], device="cuda")
    want = check_against_oracle(rt, x["logits"], x["draft"])
    # the planted prefix is a design value: where it is strictly inside the
    # block, the oracle must have found exactly it
    a = x["planted_prefix"].cpu().numpy()
    assert np.array_equal(want["accept_len"], a)


def random_case(B, K, V, dtype, seed, ties=False, device="cuda"):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    logits = torch.randn((B, K + 1, V), generator=g, device=device).to(dtype)
    draft = torch.randint(0, V, (B, K), generator=g, device=device, dtype=torch.int64)
    a = torch.randint(0, K + 1, (B,), generator=g, device=device)
    plant_prefix(logits, draft, a, ties=ties)
    return logits, draft.to(torch.int32)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize(
    "B,K,V",
    [(1, 0, 5), (1, 1, 1), (2, 1, 2), (3, 3, 7), (2, 4, 8), (2, 4, 9), (5, 16, 1023), (1, 16, 1025),
     (37, 5, 4097), (4, 40, 3001), (2, 16, 100003), (1, 16, 151936), (3, 7, 151937)],
)
def test_verify_ragged_shapes(rt, B, K, V, dtype):
    logits, draft = random_case(B, K, V, dtype, seed=B * 1000 + K * 10 + V, ties=V > 16)
    check_against_oracle(rt, logits, draft)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("V", [64, 4099, 151936])
def test_verify_dense_ties_lowest_index(rt, dtype, V):
    """Rows drawn from a 4-value set: the maximum repeats all over the row."""
    g = torch.Generator(device="cuda")
    g.manual_seed(V)
    B, K = 6, 8
    vals = torch.tensor([-1.0, 0.0, 0.5, 1.0], device="cuda")
    logits = vals[torch.randint(0, 4, (B, K + 1, V), generator=g, device="cuda")].to(dtype)
    # a few rows whose single maximum sits at the very end, or only at index 0
    logits[0, 1, :] = 0.5
    logits[0, 1, V - 1] = 1.0
    logits[1, 2, :] = 0.5
    logits[1, 2, 0] = 1.0
    draft = torch.randint(0, 2, (B, K), generator=g, device="cuda", dtype=torch.int32)
    want = check_against_oracle(rt, logits, draft)
    assert want["target_argmax"][0, 1] == V - 1 and want["target_argmax"][1, 2] == 0


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_verify_signed_zero_equal_and_infinite_rows(rt, dtype):
    V, K = 3000, 5
    logits = torch.randn((1, K + 1, V), device="cuda").to(dtype)
    logits[0, 0] = -0.0
    logits[0, 0, 17] = 0.0  # +0 after -0's: the first (a -0) wins
    logits[0, 1] = -1.0
    logits[0, 1, 2999] = -0.0
    logits[0, 1, 5] = 0.0  # +0 at 5 and -0 at 2999 tie: 5 wins
    logits[0, 2] = 3.0  # all equal: index 0
    logits[0, 3] = float("-inf")  # all -inf: index 0
    logits[0, 4] = float("-inf")
    logits[0, 4, 1234] = -1e30 if dtype == torch.float32 else -1e30
    draft = torch.tensor([[0, 5, 0, 0, 1234]], dtype=torch.int32, device="cuda")
    want = check_against_oracle(rt, logits, draft)
    assert list(want["target_argmax"][0, :5]) == [0, 5, 0, 0, 1234]
    assert want["accept_len"][0] == 5


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("pad", [3, 8, 64])
def test_verify_strided_logits(rt, dtype, pad):
    """Rows and sequences with gaps (aligned and unaligned row strides)."""
    B, K, V = 4, 6, 5000
    big_logits, draft = random_case(B, K + 2, V + pad, dtype, seed=pad)
    logits = big_logits[:, : K + 1, :V]  # row stride V + pad, batch stride (K+3)*(V+pad)
    assert logits.stride(1) == V + pad
    check_against_oracle(rt, logits, draft[:, :K].contiguous())


def test_verify_out_of_range_draft_never_matches(rt):
    B, K, V = 3, 4, 777
    logits, draft = random_case(B, K, V, torch.bfloat16, seed=3)
    targ = oracle.target_argmax(host_f64(logits))
    d = torch.from_numpy(targ[:, :K].astype(np.int32)).cuda()  # would accept everything
    d[0, 0] = -1
    d[1, 2] = V
    d[2, 3] = 2 ** 31 - 1
    want = check_against_oracle(rt, logits, d)
    assert list(want["accept_len"]) == [0, 2, 3]


def test_verify_repeatable_and_workspace_reusable(rt):
    """Ten calls, shapes changing between them, on one workspace: identical results.

    The split reductions fold per-CTA keys with atomics and a last-arriver
    ticket; a race or a key/ticket left behind by one call would show up as
    a difference here."""
    ws = rt.Workspace(64, 16, 151936, 8, torch.bfloat16)
    cases = [random_case(64, 16, 151936, torch.bfloat16, seed=s, ties=True) for s in (1, 2)]
    small = random_case(3, 5, 999, torch.bfloat16, seed=9)
    ref = [run_verify(rt, *c, ws=ws) for c in cases]
    for it in range(10):
        run_verify(rt, *small, ws=ws)
        c = it % 2
        got = run_verify(rt, *cases[c], ws=ws)
        for a, b in zip(got, ref[c]):
            assert torch.equal(a, b)
    assert ws.check() == 0


def test_verify_empty_batch(rt):
    ws = rt.Workspace(1, 4, 10, 8, torch.bfloat16)
    logits = torch.empty((0, 5, 10), dtype=torch.bfloat16, device="cuda")
    z = torch.empty((0,), dtype=torch.int32, device="cuda")
    rt.retrace_verify(logits, torch.empty((0, 4), dtype=torch.int32, device="cuda"), z,
                      torch.empty((0, 5), dtype=torch.int32, device="cuda"), z, ws)
    torch.cuda.synchronize()
