"""Pins of the CPU oracle against facts fixed outside it (no GPU).

Each test checks the oracle against something other than itself: the
paper's Fig. 3 worked example, brute force on tiny inputs (tests/brute_force.py,
which takes different routes: a stable sort for the argmax, a search over
every candidate accepted length, explicit split sums for the projections),
closed forms (closed gate, zero correction, half-open gate), invariants of
prefix verification, and an independent bf16 conversion (torch's).
``test_planted_mistakes_are_caught`` plants plausible mistakes in the oracle
and checks that these pins fail on each.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

import brute_force as bf
import oracle
from oracle import retrace_oracle as orc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# bfloat16 format
# ---------------------------------------------------------------------------


def test_bf16_decode_matches_torch_on_every_pattern():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.bf16_bits_to_f64(bits)
    ref = torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).double().numpy()
    finite = np.isfinite(ref)
    assert np.array_equal(ours[finite], ref[finite])
    assert np.array_equal(np.isnan(ours), np.isnan(ref))


def test_round_to_bf16_known_values():
    h = 2.0 ** -8  # half an ulp of bf16 at 1.0
    cases = [
        (1.0, 1.0),
        (1.0 + h, 1.0),  # tie -> even (1.0)
        (1.0 + 3 * h, 1.0 + 4 * h),  # tie -> even (1 + 2^-6)
        (1.0 + h + 2.0 ** -30, 1.0 + 2 * h),  # just above the tie -> up
        (-(1.0 + h), -1.0),
        (2.0 ** -133, 2.0 ** -133),  # smallest subnormal
        (2.0 ** -134, 0.0),  # tie between 0 and 2^-133 -> even (0)
        (3 * 2.0 ** -134, 2.0 ** -132),  # 1.5 quanta -> 2 quanta
        (255.0 * 2.0 ** 120, 255.0 * 2.0 ** 120),  # largest finite
        (2.0 ** 128 * (1 - 2.0 ** -9), math.inf),  # tie at the top -> rounds up to overflow
        (0.0, 0.0),
    ]
    for x, want in cases:
        got = oracle.round_to_bf16(np.array([x]))[0]
        assert got == want, (x, got, want)


def test_round_to_bf16_matches_torch_float32_conversion():
    # torch rounds binary32 -> bf16 to nearest even; on binary32 inputs the
    # oracle's float64 rounding must agree exactly.
    rng = np.random.default_rng(7)
    x32 = (rng.standard_normal(200_000) * np.exp(rng.uniform(-20, 20, 200_000))).astype(np.float32)
    ref = torch.from_numpy(x32).to(torch.bfloat16).double().numpy()
    ours = oracle.round_to_bf16(x32.astype(np.float64))
    assert np.array_equal(ours, ref)


def test_bf16_ulp_is_the_spacing_torch_gives():
    """bf16_ulp(x) sets the bf16 output tolerance where |reference| >= 4.  It
    must be the distance from x's bf16 interval floor to the next bf16 value:
    taken here from torch's decoding of consecutive bit patterns, over every
    positive finite pattern (zero, subnormals, every binade up to the largest
    finite value), for those values negated, and for points strictly inside
    each interval."""
    bits = np.arange(0, 0x7F7F, dtype=np.int32)  # 0x7F7F is the largest finite bf16
    lo = torch.from_numpy(bits.astype(np.int16)).view(torch.bfloat16).double().numpy()
    hi = torch.from_numpy((bits + 1).astype(np.int16)).view(torch.bfloat16).double().numpy()
    spacing = hi - lo
    assert np.array_equal(oracle.bf16_ulp(lo), spacing)
    assert np.array_equal(oracle.bf16_ulp(-lo), spacing)
    inside = lo + 0.5 * spacing  # exact in float64: both ends are bf16 values
    assert np.array_equal(oracle.bf16_ulp(inside), spacing)
    # the tolerance band the GPU tests use: 2^-5 in [4, 8), 2^-4 in [8, 16)
    assert oracle.bf16_ulp(np.array([4.0, 7.99, 8.0, 15.9]))[[0, 1, 2, 3]].tolist() == [2**-5, 2**-5, 2**-4, 2**-4]


# ---------------------------------------------------------------------------
# Verification
# ---------------------------------------------------------------------------


def test_argmax_lowest_index_on_ties_brute_force():
    rng = np.random.default_rng(1)
    values = np.array([-1.0, -0.0, 0.0, 0.5, 1.0, 1.0])
    for _ in range(400):
        K1 = int(rng.integers(1, 5))
        V = int(rng.integers(1, 40))
        logits = rng.choice(values, size=(1, K1, V))
        t = oracle.target_argmax(logits)[0]
        for i in range(K1):
            assert t[i] == bf.argmax_by_sort(list(logits[0, i])), (logits[0, i], t[i])


def test_argmax_signed_zero_and_all_equal_rows():
    row = np.array([[[-0.0, 0.0, -0.0, -1.0], [-3.0, -3.0, -3.0, -3.0]]])
    assert list(oracle.target_argmax(row)[0]) == [0, 0]
    neg_inf = np.full((1, 1, 5), -np.inf)
    assert oracle.target_argmax(neg_inf)[0, 0] == 0


def test_accept_len_brute_force():
    rng = np.random.default_rng(2)
    for _ in range(500):
        K = int(rng.integers(0, 9))
        t = rng.integers(0, 3, size=(1, K + 1))
        draft = rng.integers(0, 3, size=(1, K))
        assert oracle.accepted_length(t, draft)[0] == bf.accept_len_by_search(list(t[0]), list(draft[0]))


def test_verification_invariants():
    """Rejected tokens are never committed; committed = target-argmax prefix + bonus."""
    rng = np.random.default_rng(3)
    for _ in range(300):
        B, K, V = int(rng.integers(1, 4)), int(rng.integers(1, 8)), int(rng.integers(2, 6))
        logits = rng.integers(-2, 3, size=(B, K + 1, V)).astype(np.float64)
        draft = rng.integers(-1, V + 1, size=(B, K))  # includes out-of-range tokens
        out = oracle.verify(logits, draft)
        t, A, committed, bonus = out["target_argmax"], out["accept_len"], out["committed"], out["bonus"]
        for b in range(B):
            a = int(A[b])
            assert 0 <= a <= K
            # committed tokens are exactly the target's choices up to and including slot A
            assert list(committed[b, : a + 1]) == list(t[b, : a + 1])
            assert list(committed[b, :a]) == list(draft[b, :a])
            assert all(x == -1 for x in committed[b, a + 1 :])
            assert bonus[b] == t[b, a]
            if a < K:  # the first rejected draft token is not what gets committed there
                assert committed[b, a] != draft[b, a]
            # out-of-range draft tokens can never be accepted
            for i in range(a):
                assert 0 <= draft[b, i] < V


def _fig3():
    with open(os.path.join(GOLDEN, "fig3_worked_example.json")) as f:
        fx = json.load(f)
    vocab = fx["vocab"]
    tok = {w: i for i, w in enumerate(vocab)}
    return fx, vocab, tok


@pytest.mark.parametrize("unstated_choice", ["<unstated>", "but", ",", "he"])
def test_fig3_worked_example(unstated_choice):
    fx, vocab, tok = _fig3()
    K, V, d = len(fx["draft"]), len(vocab), 3
    draft = np.array([[tok[w] for w in fx["draft"]]])
    logits = np.zeros((1, K + 1, V))
    for i, w in enumerate(fx["target_choice_per_slot"]):
        logits[0, i, tok[unstated_choice if w == "<unstated>" else w]] = 1.0
    out = oracle.verify(logits, draft)
    exp = fx["expected"]
    A = int(out["accept_len"][0])
    assert A == exp["accept_len"]
    assert A + 1 == exp["first_rejected_slot_paper_1based"]
    assert [vocab[x] for x in out["committed"][0, : A + 1]] == exp["committed"]
    assert vocab[out["bonus"][0]] == exp["correction_token"]
    n = oracle.carried_rows(out["accept_len"], K)
    assert int(n[0]) == exp["carried_rows"]
    # hD row k encodes the draft token of slot k; the carried rows must be the
    # states of the rejected suffix "but he", shifted to the block start.
    hD = np.zeros((1, K, d))
    for k in range(K):
        hD[0, k, 0] = draft[0, k]
    hT = np.zeros((1, K, d))
    m, _ = oracle.align(hD, hT, out["accept_len"])
    carried = [vocab[int(m[0, j, 0])] for j in range(int(n[0]))]
    assert carried == exp["carried_draft_tokens"]
    assert not m[0, int(n[0]) :].any()


def test_reset_rule_and_initial_state():
    K = 6
    A = np.array([0, 1, K - 2, K - 1, K])
    assert list(oracle.carried_rows(A, K)) == [K - 1, K - 2, 1, 0, 0]


def test_align_pairs_draft_and_target_states_of_the_same_slot():
    """u_j is the target state whose logits score the slot that m_j drafted (Eq. 5)."""
    rng = np.random.default_rng(4)
    for _ in range(50):
        B, K, d = 3, int(rng.integers(1, 9)), 2
        A = rng.integers(0, K + 1, size=B)
        hD = np.zeros((B, K, d))
        hT = np.zeros((B, K, d))
        for k in range(K):
            hD[:, k, 0] = k + 1  # drafter state of slot k (label = slot + 1)
            hT[:, k, 0] = k + 2  # target state at slot k scores slot k + 1
        m, u = oracle.align(hD, hT, A)
        n = oracle.carried_rows(A, K)
        for b in range(B):
            for j in range(K):
                if j < n[b]:
                    assert m[b, j, 0] == u[b, j, 0] == A[b] + 1 + j + 1
                else:
                    assert m[b, j, 0] == u[b, j, 0] == 0


# ---------------------------------------------------------------------------
# Projections and gate: brute force and closed forms
# ---------------------------------------------------------------------------


def _tiny(rng, B, K, V, d):
    logits = rng.standard_normal((B, K + 1, V))
    draft = rng.integers(0, V, size=(B, K))
    for b in range(B):  # plant an accepted prefix so the suffix is exercised
        a = int(rng.integers(0, K + 1))
        for i in range(a):
            logits[b, i, draft[b, i]] = logits[b, i].max() + 1
    return dict(
        logits=logits,
        draft=draft,
        hD=rng.standard_normal((B, K, d)),
        hT=rng.standard_normal((B, K, d)),
        e=rng.standard_normal((B, K, d)) * 0.1,
        Wc=rng.standard_normal((d, 2 * d)) / math.sqrt(d),
        Wv=rng.standard_normal((d, d)) / math.sqrt(d),
        Wg=rng.standard_normal((d, 2 * d)) / math.sqrt(d),
        beta=float(rng.uniform(0.25, 1.5)),
    )


def _check_round_against_brute(x, dtype="f32"):
    out = oracle.retrace_round(
        x["logits"], x["draft"], x["hD"], x["hT"], x["e"], x["Wc"], x["Wv"], x["Wg"], x["beta"], dtype
    )
    B, K = x["draft"].shape
    rnd = (lambda r: list(oracle.round_to_bf16(np.array(r)))) if dtype == "bf16" else None
    for b in range(B):
        ref = bf.round_brute(
            x["logits"][b].tolist(),
            x["draft"][b].tolist(),
            x["hD"][b].tolist(),
            x["hT"][b].tolist(),
            x["e"][b].tolist(),
            x["Wc"].tolist(),
            x["Wv"].tolist(),
            x["Wg"].tolist(),
            x["beta"],
            rnd=rnd,
        )
        assert list(out["target_argmax"][b]) == ref["t"]
        assert out["accept_len"][b] == ref["A"]
        assert list(out["committed"][b, : ref["A"] + 1]) == ref["committed"]
        assert out["bonus"][b] == ref["bonus"]
        assert out["n"][b] == ref["n"]
        np.testing.assert_allclose(out["e_tilde"][b], np.array(ref["e_tilde"]), rtol=1e-12, atol=1e-12)


def test_round_brute_force_random_tiny_shapes():
    rng = np.random.default_rng(5)
    for _ in range(150):
        B, K, V, d = int(rng.integers(1, 3)), int(rng.integers(1, 9)), int(rng.integers(1, 65)), int(rng.integers(1, 9))
        _check_round_against_brute(_tiny(rng, B, K, V, d))


def test_round_brute_force_bf16_rounding_point():
    rng = np.random.default_rng(6)
    for _ in range(40):
        _check_round_against_brute(_tiny(rng, 2, 5, 16, 6), dtype="bf16")


def test_closed_gate_reproduces_mask_input_exactly():
    """W_v = 0 (the paper's initialisation) gives e~ = e bit-for-bit."""
    rng = np.random.default_rng(8)
    x = _tiny(rng, 3, 6, 20, 8)
    x["Wv"] = np.zeros_like(x["Wv"])
    out = oracle.retrace_round(**{k: x[k] for k in ("logits", "draft", "hD", "hT", "e", "Wc", "Wv", "Wg", "beta")}, dtype="f32")
    assert np.array_equal(out["e_tilde"], x["e"])


def test_half_open_gate_and_identity_value_projection():
    """W_g = 0 gives sigmoid = 1/2; with W_v = I and beta = 0: e~ = e + m/2 exactly."""
    rng = np.random.default_rng(9)
    B, K, d = 2, 7, 5
    x = _tiny(rng, B, K, 12, d)
    x["Wg"] = np.zeros_like(x["Wg"])
    x["Wv"] = np.eye(d)
    x["beta"] = 0.0
    out = oracle.retrace_round(**{k: x[k] for k in ("logits", "draft", "hD", "hT", "e", "Wc", "Wv", "Wg", "beta")}, dtype="f32")
    A, n = out["accept_len"], out["n"]
    for b in range(B):
        for j in range(K):
            if j < n[b]:
                want = x["e"][b, j] + 0.5 * x["hD"][b, A[b] + 1 + j]
            else:
                want = x["e"][b, j]
            assert np.array_equal(out["e_tilde"][b, j], want)


def test_zero_correction_keeps_the_aligned_draft_state():
    """W_c = 0 (or beta = 0) gives r = m (Eq. 7)."""
    rng = np.random.default_rng(10)
    x = _tiny(rng, 2, 6, 10, 4)
    A = oracle.verify(x["logits"], x["draft"])["accept_len"]
    m, u = oracle.align(x["hD"], x["hT"], A)
    assert np.array_equal(oracle.correct(m, u, np.zeros_like(x["Wc"]), 1.0, False), m)
    assert np.array_equal(oracle.correct(m, u, x["Wc"], 0.0, False), m)


def test_sigmoid_reference_values():
    z = np.array([0.0, 1.0, -1.0, 40.0, -40.0, -800.0, 800.0])
    want = np.array([0.5, 1 / (1 + math.exp(-1)), math.exp(-1) / (1 + math.exp(-1)), 1 / (1 + math.exp(-40)),
                     math.exp(-40) / (1 + math.exp(-40)), 0.0, 1.0])
    np.testing.assert_allclose(oracle.sigmoid(z), want, rtol=1e-15, atol=0)


def test_conditioned_rows_agree_with_full_round():
    rng = np.random.default_rng(11)
    x = _tiny(rng, 3, 8, 30, 6)
    e_vec = x["e"][0, 0]
    for dtype in ("f32", "bf16"):
        out = oracle.retrace_round(x["logits"], x["draft"], x["hD"], x["hT"], e_vec, x["Wc"], x["Wv"], x["Wg"], x["beta"], dtype)
        rows = [(b, j) for b in range(3) for j in range(8)]
        got = oracle.conditioned_rows(rows, out["accept_len"], x["hD"], x["hT"], e_vec, x["Wc"], x["Wv"], x["Wg"], x["beta"], dtype)
        full = out["e_tilde_rounded"] if dtype == "bf16" else out["e_tilde"]
        np.testing.assert_allclose(got, full.reshape(-1, 6), rtol=1e-13, atol=1e-13)


# ---------------------------------------------------------------------------
# Ablation variants (Sec. "Component Ablation", Table 3; Appendix "Ablation
# Settings"): the same aligned signal, used three other ways
# ---------------------------------------------------------------------------


def test_fig3_overwrite_carries_the_rejected_suffix():
    """Overwrite: the next block starts with the drafter states of "but he"
    (Fig. 3) in place of the mask inputs; the other positions keep e."""
    fx, vocab, tok = _fig3()
    K, V, d = len(fx["draft"]), len(vocab), 3
    draft = np.array([[tok[w] for w in fx["draft"]]])
    logits = np.zeros((1, K + 1, V))
    for i, w in enumerate(fx["target_choice_per_slot"]):
        logits[0, i, tok["<unstated>" if w == "<unstated>" else w]] = 1.0
    hD = np.zeros((1, K, d))
    for k in range(K):
        hD[0, k] = [draft[0, k], 10.0 + k, -0.5 * k]  # label, slot, a third distinct value
    hT = np.full((1, K, d), 7.0)
    e_vec = np.array([-1.0, -2.0, -3.0])
    out = oracle.retrace_round(logits, draft, hD, hT, e_vec, None, None, None, 1.0, "f32", variant="overwrite")
    n = fx["expected"]["carried_rows"]
    assert int(out["n"][0]) == n
    assert [vocab[int(out["e_tilde"][0, j, 0])] for j in range(n)] == fx["expected"]["carried_draft_tokens"]
    A = fx["expected"]["accept_len"]
    for j in range(n):  # the whole state row of slot A+1+j, bit for bit
        assert np.array_equal(out["e_tilde"][0, j], hD[0, A + 1 + j])
    assert np.array_equal(out["e_tilde"][0, n:], np.broadcast_to(e_vec, (K - n, d)))


def _brute_rows(x, b, beta):
    return bf.round_brute(x["logits"][b].tolist(), x["draft"][b].tolist(), x["hD"][b].tolist(), x["hT"][b].tolist(),
                          x["e"][b].tolist(), x["Wc"].tolist(), x["Wv"].tolist(), x["Wg"].tolist(), beta)


def test_raw_is_the_gated_fusion_of_the_aligned_draft_states():
    """Raw conditioning, gated: Eq. 8 with r = m, which is the brute-force
    round at beta = 0 (there r = m + 0 * c = m exactly).  The oracle is given
    a non-zero beta, which the raw variant must ignore."""
    rng = np.random.default_rng(21)
    for B, K, V, d in [(3, 5, 11, 4), (2, 8, 7, 3), (4, 2, 5, 2)]:
        x = _tiny(rng, B, K, V, d)
        out = oracle.retrace_round(x["logits"], x["draft"], x["hD"], x["hT"], x["e"], x["Wc"], x["Wv"], x["Wg"],
                                   x["beta"], "f32", variant="raw")
        for b in range(B):
            want = _brute_rows(x, b, 0.0)
            assert int(out["n"][b]) == want["n"]
            np.testing.assert_allclose(out["e_tilde"][b], np.array(want["e_tilde"]), rtol=1e-12, atol=1e-12)
        corrected = oracle.retrace_round(x["logits"], x["draft"], x["hD"], x["hT"], x["e"], x["Wc"], x["Wv"],
                                         x["Wg"], x["beta"], "f32")
        if int(out["n"].sum()) > 0:  # the correction changes something where rows are carried
            assert not np.allclose(out["e_tilde"], corrected["e_tilde"])


def test_none_keeps_every_input_and_still_reports_n():
    """No conditioning (the DFlash row): e~ = e everywhere; n_b is still the
    carried-row count of the verification."""
    rng = np.random.default_rng(22)
    x = _tiny(rng, 4, 6, 9, 3)
    out = oracle.retrace_round(x["logits"], x["draft"], x["hD"], x["hT"], x["e"], None, None, None, x["beta"],
                               "bf16", variant="none")
    assert np.array_equal(out["e_tilde"], x["e"])
    assert [int(v) for v in out["n"]] == [_brute_rows(x, b, x["beta"])["n"] for b in range(4)]


# ---------------------------------------------------------------------------
# Low-rank realisation (Appendix "Concurrent-Serving Experiment")
# ---------------------------------------------------------------------------


def _tiny_lowrank(rng, B, K, V, d, L, C):
    x = _tiny(rng, B, K, V, d)
    x.update(
        P=rng.standard_normal((L, d)) / math.sqrt(d),
        Bc=rng.standard_normal((C, L + d)) / math.sqrt(L + d),
        Ac=rng.standard_normal((L, C)) / math.sqrt(C),
        Wv=rng.standard_normal((d, L)) / math.sqrt(L),
        Wg=rng.standard_normal((d, d + L)) / math.sqrt(d + L),
    )
    return x


def _check_lowrank_against_brute(x, dtype="f32"):
    out = oracle.retrace_round_lowrank(x["logits"], x["draft"], x["hD"], x["hT"], x["e"], x["P"], x["Bc"], x["Ac"],
                                       x["Wv"], x["Wg"], x["beta"], dtype)
    rnd = (lambda r: list(oracle.round_to_bf16(np.array(r)))) if dtype == "bf16" else None
    for b in range(x["draft"].shape[0]):
        ref = bf.lowrank_brute(x["logits"][b].tolist(), x["draft"][b].tolist(), x["hD"][b].tolist(),
                               x["hT"][b].tolist(), x["e"][b].tolist(), x["P"].tolist(), x["Bc"].tolist(),
                               x["Ac"].tolist(), x["Wv"].tolist(), x["Wg"].tolist(), x["beta"], rnd=rnd)
        assert out["accept_len"][b] == ref["A"] and out["n"][b] == ref["n"]
        np.testing.assert_allclose(out["e_tilde"][b], np.array(ref["e_tilde"]), rtol=1e-12, atol=1e-12)


def test_lowrank_brute_force_random_tiny_shapes():
    rng = np.random.default_rng(31)
    for _ in range(60):
        B, K, V, d = int(rng.integers(1, 3)), int(rng.integers(1, 8)), int(rng.integers(2, 40)), int(rng.integers(1, 7))
        L, C = int(rng.integers(1, 5)), int(rng.integers(1, 4))
        _check_lowrank_against_brute(_tiny_lowrank(rng, B, K, V, d, L, C))


def test_lowrank_brute_force_bf16_rounding_points():
    rng = np.random.default_rng(32)
    for _ in range(30):
        _check_lowrank_against_brute(_tiny_lowrank(rng, 2, 6, 16, 5, 3, 2), dtype="bf16")


def test_lowrank_with_a_full_width_latent_is_the_method():
    """With the latent as wide as the state (L = d) and P = I, the low-rank
    path is Eq. 6-8 with W_c = A_c B_c (a rank-C correction), the value and
    gate projections unchanged: the brute-force method round must agree."""
    rng = np.random.default_rng(33)
    for _ in range(20):
        d, C = int(rng.integers(2, 6)), int(rng.integers(1, 4))
        x = _tiny_lowrank(rng, 2, 6, 12, d, d, C)
        x["P"] = np.eye(d)
        Wc = x["Ac"] @ x["Bc"]  # [d, 2d]
        for dtype in ("f32", "bf16"):
            # bf16: the latent z = m is then exact (m holds bf16 values), and
            # both paths round the same corrected value once
            hD = oracle.round_to_bf16(x["hD"]) if dtype == "bf16" else x["hD"]
            out = oracle.retrace_round_lowrank(x["logits"], x["draft"], hD, x["hT"], x["e"], x["P"], x["Bc"],
                                               x["Ac"], x["Wv"], x["Wg"], x["beta"], dtype)
            rnd = (lambda r: list(oracle.round_to_bf16(np.array(r)))) if dtype == "bf16" else None
            for b in range(2):
                ref = bf.round_brute(x["logits"][b].tolist(), x["draft"][b].tolist(), hD[b].tolist(),
                                     x["hT"][b].tolist(), x["e"][b].tolist(), Wc.tolist(), x["Wv"].tolist(),
                                     x["Wg"].tolist(), x["beta"], rnd=rnd)
                np.testing.assert_allclose(out["e_tilde"][b], np.array(ref["e_tilde"]), rtol=1e-11, atol=1e-11)


# ---------------------------------------------------------------------------
# Stochastic verification (speculative sampling on filtered distributions)
# ---------------------------------------------------------------------------


def _sampled_case(rng, B, K, V, spread=1.5):
    tl = rng.standard_normal((B, K + 1, V)) * spread
    dl = tl[:, :K] + rng.standard_normal((B, K, V)) * 0.7  # a drafter close to the target
    draft = np.argsort(-dl, axis=-1, kind="stable")[:, :, :3][np.arange(B)[:, None], np.arange(K)[None, :],
                                                              rng.integers(0, 3, size=(B, K))]
    return tl, dl, draft, rng.random((B, K + 1))


def test_filtered_distribution_brute_force():
    rng = np.random.default_rng(41)
    for _ in range(200):
        V = int(rng.integers(1, 30))
        row = np.round(rng.standard_normal(V) * 2, 1)  # rounding plants equal logits
        T, k, pth = float(rng.uniform(0.3, 2.0)), int(rng.integers(1, V + 1)), float(rng.uniform(0.05, 1.0))
        toks, probs = oracle.filtered_distribution(row, T, k, pth)
        bt, bp = bf.filtered_brute(row.tolist(), T, k, pth)
        assert list(toks) == bt
        np.testing.assert_allclose(probs, bp, rtol=1e-12, atol=1e-14)


def test_sampled_verification_brute_force():
    rng = np.random.default_rng(42)
    for _ in range(40):
        B, K, V = int(rng.integers(1, 4)), int(rng.integers(1, 7)), int(rng.integers(2, 25))
        T, k, pth = float(rng.uniform(0.5, 1.5)), int(rng.integers(1, V + 1)), float(rng.uniform(0.5, 1.0))
        tl, dl, draft, u = _sampled_case(rng, B, K, V)
        out = oracle.verify_sampled(tl, dl, draft, u, T, k, pth)
        for b in range(B):
            ref = bf.sampled_brute(tl[b].tolist(), dl[b].tolist(), draft[b].tolist(), u[b].tolist(), T, k, pth)
            assert out["accept_len"][b] == ref["A"]
            assert list(out["committed"][b, : ref["A"] + 1]) == ref["committed"]


def test_sampled_verification_is_lossless():
    """The defining property: over the random numbers, the first committed
    token is distributed as the filtered target distribution p_0, whatever the
    draft token and the draft distribution (integrated over a fine grid of
    (u_0, u_K) here, exact up to the grid)."""
    rng = np.random.default_rng(43)
    V, T, k, pth = 7, 1.0, 5, 0.9
    N = 400
    grid = (np.arange(N) + 0.5) / N
    for _ in range(3):
        tl = rng.standard_normal((1, 2, V)) * 1.5
        dl = rng.standard_normal((1, 1, V)) * 1.5
        qt, qp = oracle.filtered_distribution(dl[0, 0], T, k, pth)
        pt, pp = oracle.filtered_distribution(tl[0, 0], T, k, pth)
        want = np.zeros(V)
        want[pt] = pp
        got = np.zeros(V)
        for x, qx in zip(qt, qp):  # the draft token is drawn from q
            for u0 in grid:
                for uk in grid[::8]:
                    y = oracle.verify_sampled(tl, dl, np.array([[x]]), np.array([[u0, uk]]), T, k, pth)["committed"][0, 0]
                    got[y] += qx / (N * len(grid[::8]))
        np.testing.assert_allclose(got, want, atol=3e-2)


def test_sampled_verification_with_top_k_one_is_greedy():
    """top_k = 1 makes both distributions one-hot on the row argmax, so with
    drafts equal to the drafter's argmax the block is verified exactly as by
    greedy verification, for any random numbers."""
    rng = np.random.default_rng(44)
    for _ in range(20):
        B, K, V = 3, 6, 17
        tl = rng.standard_normal((B, K + 1, V))
        dl = tl[:, :K] + rng.standard_normal((B, K, V)) * 0.6
        draft = np.argmax(dl, axis=-1)
        out = oracle.verify_sampled(tl, dl, draft, rng.random((B, K + 1)), 1.0, 1, 0.95)
        ref = oracle.verify(tl, draft)
        np.testing.assert_array_equal(out["accept_len"], ref["accept_len"])
        np.testing.assert_array_equal(out["committed"], ref["committed"])


def test_sampled_verification_accepts_everything_when_draft_equals_target():
    """q = p and drafts drawn from it: u q(x) < p(x) = q(x) holds for every
    u < 1, so the whole block is accepted and the bonus comes from p_K."""
    rng = np.random.default_rng(45)
    B, K, V = 4, 5, 11
    tl = rng.standard_normal((B, K + 1, V))
    draft = np.argsort(-tl[:, :K], axis=-1, kind="stable")[:, :, 0]
    out = oracle.verify_sampled(tl, tl[:, :K].copy(), draft, rng.random((B, K + 1)), 1.0, 4, 0.9)
    assert (out["accept_len"] == K).all()


# ---------------------------------------------------------------------------
# Planted mistakes: every one must make at least one pin above fail
# ---------------------------------------------------------------------------


def _pins():
    return [
        test_argmax_lowest_index_on_ties_brute_force,
        test_accept_len_brute_force,
        lambda: test_fig3_worked_example("<unstated>"),
        test_reset_rule_and_initial_state,
        test_align_pairs_draft_and_target_states_of_the_same_slot,
        test_round_brute_force_random_tiny_shapes,
        test_closed_gate_reproduces_mask_input_exactly,
        test_half_open_gate_and_identity_value_projection,
        test_zero_correction_keeps_the_aligned_draft_state,
        test_sigmoid_reference_values,
        test_fig3_overwrite_carries_the_rejected_suffix,
        test_raw_is_the_gated_fusion_of_the_aligned_draft_states,
        test_none_keeps_every_input_and_still_reports_n,
        test_lowrank_brute_force_random_tiny_shapes,
        test_lowrank_brute_force_bf16_rounding_points,
        test_lowrank_with_a_full_width_latent_is_the_method,
        test_filtered_distribution_brute_force,
        test_sampled_verification_brute_force,
        test_sampled_verification_with_top_k_one_is_greedy,
        test_sampled_verification_accepts_everything_when_draft_equals_target,
        test_bf16_ulp_is_the_spacing_torch_gives,
    ]


def _mut_ulp_below(x):
    a = np.abs(np.asarray(x, dtype=np.float64))
    mant, _ = np.frexp(a)
    return orc.__dict__["_orig_bf16_ulp"](x) * np.where(mant == 0.5, 0.5, 1.0)


def _mut_argmax_last(logits):
    lg = np.asarray(logits, dtype=np.float64)
    return (lg.shape[-1] - 1 - np.argmax(lg[..., ::-1], axis=-1)).astype(np.int64)


def _mut_align_u_shift(hD, hT, A):
    hD = np.asarray(hD, float)
    hT = np.asarray(hT, float)
    B, K, d = hD.shape
    n = orc.carried_rows(A, K)
    m = np.zeros_like(hD)
    u = np.zeros_like(hT)
    for b in range(B):
        for j in range(int(n[b])):
            m[b, j] = hD[b, A[b] + 1 + j]
            u[b, j] = hT[b, min(A[b] + 1 + j, K - 1)]  # off by one: hT of the drafted slot
    return m, u


def _mut_align_keep_rejected(hD, hT, A):
    hD = np.asarray(hD, float)
    hT = np.asarray(hT, float)
    B, K, d = hD.shape
    n = orc.carried_rows(A, K)
    m = np.zeros_like(hD)
    u = np.zeros_like(hT)
    for b in range(B):
        for j in range(int(n[b])):
            m[b, j] = hD[b, A[b] + j]  # includes the first rejected slot
            u[b, j] = hT[b, A[b] + j]
    return m, u


def _mut_condition(change):
    def f(e_full, m, u, n, Wc, Wv, Wg, beta, variant, rr):
        return orc.__dict__["_orig_condition"](e_full, m, u, n, Wc, Wv, Wg, beta, change.get(variant, variant), rr)
    return f


def _mut_overwrite_unshifted(e_full, m, u, n, Wc, Wv, Wg, beta, variant, rr):
    if variant != "overwrite":
        return orc.__dict__["_orig_condition"](e_full, m, u, n, Wc, Wv, Wg, beta, variant, rr)
    K = m.shape[1]
    rows = np.arange(K)[None, :] < np.asarray(n)[:, None]
    shifted = np.concatenate([m[:, -1:], m[:, :-1]], axis=1)  # rows land one position late
    return None, np.where(rows[..., None], shifted, e_full)


def _mut_lowrank(**change):
    def f(e_full, m, u, n, P, Bc, Ac, Wv, Wg, beta, round_bf16):
        args = dict(e_full=e_full, m=m, u=u, n=n, P=P, Bc=Bc, Ac=Ac, Wv=Wv, Wg=Wg, beta=beta, round_bf16=round_bf16)
        for k, fn in change.items():
            args[k] = fn(args)
        return orc.__dict__["_orig_lowrank"](**args)
    return f


def _mut_lowrank_swapped_halves(e_full, m, u, n, P, Bc, Ac, Wv, Wg, beta, round_bf16):
    L = np.asarray(P).shape[0]
    d = np.asarray(m).shape[-1]
    Bc = np.asarray(Bc)
    # B_c applied to [u; z] instead of [z; u]: the first d columns act on u
    swapped = np.concatenate([Bc[:, d:], Bc[:, :d]], axis=1) if Bc.shape[1] == L + d and L != d else Bc[:, ::-1]
    return orc.__dict__["_orig_lowrank"](e_full, m, u, n, P, swapped, Ac, Wv, Wg, beta, round_bf16)


def _mut_filtered(kind):
    def f(logits_row, T, top_k, top_p):
        if kind == "no_temperature":
            return orc.__dict__["_orig_filtered"](logits_row, 1.0, top_k, top_p)
        toks, probs = orc.__dict__["_orig_filtered"](logits_row, T, top_k, 1.0)
        if kind == "top_p_drops_crossing":  # keeps only the prefix strictly below top_p
            keep = max(1, int(np.searchsorted(np.cumsum(probs), top_p, side="left")))
        else:  # top-p ignored
            keep = len(toks)
        return toks[:keep], probs[:keep] / probs[:keep].sum()
    return f


MUTATIONS = {
    "bf16 ulp exponent off by one": ("bf16_ulp", lambda x: 2.0 * orc.__dict__["_orig_bf16_ulp"](x)),
    "bf16 ulp measured below x (half at powers of two)": ("bf16_ulp", _mut_ulp_below),
    "temperature ignored": ("filtered_distribution", _mut_filtered("no_temperature")),
    "top-p drops the crossing token": ("filtered_distribution", _mut_filtered("top_p_drops_crossing")),
    "top-p ignored": ("filtered_distribution", _mut_filtered("no_top_p")),
    "low-rank correction drops beta": ("lowrank_condition", _mut_lowrank(beta=lambda a: 1.0)),
    "low-rank latent not rounded": ("lowrank_condition", _mut_lowrank(round_bf16=lambda a: False)),
    "low-rank gate ignores e": (
        "lowrank_condition",
        _mut_lowrank(Wg=lambda a: np.concatenate([np.zeros_like(np.asarray(a["Wg"])[:, : np.asarray(a["m"]).shape[-1]]),
                                                  np.asarray(a["Wg"])[:, np.asarray(a["m"]).shape[-1]:]], 1)),
    ),
    "low-rank B_c halves swapped": ("lowrank_condition", _mut_lowrank_swapped_halves),
    "overwrite keeps the mask inputs": ("condition", _mut_condition({"overwrite": "none"})),
    "raw applies the correction": ("condition", _mut_condition({"raw": "corrected"})),
    "no conditioning runs the gate": ("condition", _mut_condition({"none": "raw"})),
    "overwrite rows one position late": ("condition", _mut_overwrite_unshifted),
    "argmax picks the last maximum": ("target_argmax", _mut_argmax_last),
    "accept length counts all matches": (
        "accepted_length",
        lambda t, draft: np.array([int(np.sum(np.asarray(t)[b, : np.asarray(draft).shape[1]] == np.asarray(draft)[b])) for b in range(np.asarray(draft).shape[0])]),
    ),
    "carry kept at A = K-1": ("carried_rows", lambda A, K: np.maximum(0, K - np.asarray(A))),
    "u taken at the drafted slot": ("align", _mut_align_u_shift),
    "first rejected state carried": ("align", _mut_align_keep_rejected),
    "beta dropped": ("correct", lambda m, u, Wc, beta, rr: m + np.concatenate([m, u], -1) @ np.asarray(Wc).T),
    "W_c transposed halves": (
        "correct",
        lambda m, u, Wc, beta, rr: m + beta * np.concatenate([u, m], -1) @ np.asarray(Wc).T,
    ),
    "gate sign flipped": ("sigmoid", lambda z: 1.0 / (1.0 + np.exp(np.asarray(z, float)))),
    "W_v transposed": (
        "gate_fuse",
        lambda e, r, n, Wv, Wg: orc.__dict__["_orig_gate_fuse"](e, r, n, np.asarray(Wv).T, Wg),
    ),
    "gate ignores e": (
        "gate_fuse",
        lambda e, r, n, Wv, Wg: orc.__dict__["_orig_gate_fuse"](e, r, n, Wv, np.concatenate([np.zeros_like(np.asarray(Wg)[:, : np.asarray(Wv).shape[0]]), np.asarray(Wg)[:, np.asarray(Wv).shape[0]:]], 1)),
    ),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistakes_are_caught(name, monkeypatch):
    attr, fn = MUTATIONS[name]
    monkeypatch.setitem(orc.__dict__, "_orig_gate_fuse", orc.gate_fuse)
    monkeypatch.setitem(orc.__dict__, "_orig_condition", orc.condition)
    monkeypatch.setitem(orc.__dict__, "_orig_lowrank", orc.lowrank_condition)
    monkeypatch.setitem(orc.__dict__, "_orig_filtered", orc.filtered_distribution)
    monkeypatch.setitem(orc.__dict__, "_orig_bf16_ulp", orc.bf16_ulp)
    monkeypatch.setattr(orc, attr, fn)
    monkeypatch.setattr(oracle, attr, fn, raising=False)
    caught = 0
    for pin in _pins():
        try:
            pin()
        except Exception:  # an assertion or a crash: either way the pin notices
            caught += 1
    assert caught > 0, f"no pin detects the planted mistake: {name}"
