"""Plain CPU oracle for one ReTrace decoding round.

TEST INFRASTRUCTURE ONLY.  This module states what the GPU path must compute,
slowly and in float64, so that a reader can check it against the paper by eye.
Only the test suite (``tests/``), ``__graft_entry__.smoke()`` and the CPU
baseline / reference arm of ``bench.py`` may import or run it.  The product
path (the CUDA library and its Python binding) never calls it and shares no
code with it: no kernels, helpers, constants or pre/post-processing.

Paper: "ReTrace: Rejected-Trajectory Conditioning for Speculative Decoding".
Index conventions are 0-based; the paper is 1-based:

* ``K``: draft tokens per block (the paper's block size, written B there).
* ``logits[b, i]`` for ``i = 0..K`` is the target's verify distribution at draft
  slot ``i``; row ``K`` scores the bonus position.
* ``hD[b, k]`` is the drafter state of slot ``k`` (paper ``h^D_{t,k+1}``);
  ``hT[b, k]`` is the target state at the position of slot ``k`` (paper
  ``h^T_{t,k+1}``), whose logits score slot ``k+1``.
* ``A`` accepted drafts; the first rejected slot is ``A`` (paper ``r_t = A_t+1``).

Every floating input arrives as float64 values (bf16 inputs are first decoded
exactly with :func:`bf16_bits_to_f64`).  Where the GPU path rounds (``r`` to
bf16 before the gate projection; the output to bf16), the oracle applies the
same round-to-nearest-even at the same point, on its float64 values.

Parity status of each function (pinned by ``tests/test_oracle_pins.py``):
every function below is pinned — by brute force on tiny inputs, by the
paper's Fig. 3 worked example, or by closed forms.  The learned weight values
themselves are not pinned (the paper publishes no checkpoint); they are
seeded random inputs.
"""

from __future__ import annotations

import numpy as np

# ---------------------------------------------------------------------------
# Number formats
# ---------------------------------------------------------------------------


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bfloat16 bit patterns (uint16/int16 array) to exact float64 values.

    A bfloat16 value is the upper 16 bits of the IEEE binary32 value with the
    same sign, exponent and leading 7 mantissa bits, so shifting the pattern
    into the top half of a uint32 gives that binary32 value exactly.
    """
    u32 = np.asarray(bits).astype(np.uint16).astype(np.uint32) << np.uint32(16)
    return u32.view(np.float32).astype(np.float64)


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value, ties to even.

    bfloat16 keeps 8 significant bits (1 implicit + 7 stored) with binary32's
    exponent range.  For |x| in [2^(e-1), 2^e) the spacing of representable
    values is 2^(e-8); below the normal range (2^-126) the spacing stays at the
    subnormal quantum 2^-133.  Scaling by a power of two is exact, so rounding
    x / q to the nearest integer (numpy's rint: half to even) and scaling back
    gives the correctly rounded result.  Magnitudes that round beyond the
    largest finite bf16 (65280 * 2^112) become infinities.
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.array(x, dtype=np.float64, copy=True)
    finite = np.isfinite(x) & (x != 0.0)
    xf = x[finite]
    _, e = np.frexp(xf)  # xf = mant * 2**e with 0.5 <= |mant| < 1
    q_exp = np.maximum(e - 8, -133)
    q = np.ldexp(np.ones_like(xf), q_exp)
    y = np.rint(xf / q) * q
    max_bf16 = np.ldexp(255.0, 120)  # (2 - 2^-7) * 2^127
    y = np.where(np.abs(y) > max_bf16, np.copysign(np.inf, y), y)
    out[finite] = y
    return out


def bf16_ulp(x: np.ndarray) -> np.ndarray:
    """Spacing of bfloat16 values at |x| (one unit in the last place).

    For |x| in [2^(e-1), 2^e) the next larger bf16 value is 2^(e-8) away (8
    significant bits); below the normal range the spacing stays at the
    subnormal quantum 2^-133, which is also the spacing at 0.  Used for the
    bf16 output tolerance where |reference| >= 4.
    """
    x = np.abs(np.asarray(x, dtype=np.float64))
    _, e = np.frexp(np.where(x == 0.0, np.ldexp(1.0, -126), x))
    return np.ldexp(1.0, np.maximum(e - 8, -133))


# ---------------------------------------------------------------------------
# Greedy verification (Algorithm 1 "Verify" and commit steps)
# ---------------------------------------------------------------------------


def target_argmax(logits: np.ndarray) -> np.ndarray:
    """t[b, i] = argmax_v logits[b, i, v], the lowest index among equal maxima.

    Greedy verification uses top_k = 1 (Appendix "Evaluation Protocol"): the
    target's choice at every slot is its highest-scoring token.  np.argmax
    returns the first occurrence of the maximum, and -0.0 == +0.0 under its
    comparisons, which is the tie rule of this implementation.  Sequences are
    processed one at a time so that a [K+1, V] slice is the largest float64
    temporary.
    """
    logits = np.asarray(logits)
    B, K1, _ = logits.shape
    t = np.empty((B, K1), dtype=np.int64)
    for b in range(B):
        t[b] = np.argmax(np.asarray(logits[b], dtype=np.float64), axis=-1)
    return t


def accepted_length(t: np.ndarray, draft: np.ndarray) -> np.ndarray:
    """A_b: number of leading draft tokens equal to the target's choice.

    Prefix verification accepts drafts up to the first mismatch and discards
    the rest (Sec. 1; Sec. 4, "Rejected-Trajectory Construction").  A_b is the
    first slot i < K with t[b, i] != draft[b, i], or K if every draft matches.
    """
    t = np.asarray(t)
    draft = np.asarray(draft)
    B, K = draft.shape
    A = np.full(B, K, dtype=np.int64)
    for b in range(B):
        for i in range(K):
            if t[b, i] != draft[b, i]:
                A[b] = i
                break
    return A


def commit(t: np.ndarray, draft: np.ndarray, A: np.ndarray):
    """Tokens appended to the context this round (Algorithm 1, commit step).

    The A_b accepted drafts are appended, then the target's own token at slot
    A_b: the correction token when A_b < K, the bonus token when the whole
    block was accepted.  Returns ``committed`` [B, K+1] (unused tail = -1) and
    ``bonus`` [B] (= the token at slot A_b).
    """
    t = np.asarray(t)
    draft = np.asarray(draft)
    B, K = draft.shape
    committed = np.full((B, K + 1), -1, dtype=np.int64)
    bonus = np.empty(B, dtype=np.int64)
    for b in range(B):
        a = int(A[b])
        committed[b, :a] = draft[b, :a]
        committed[b, a] = t[b, a]
        bonus[b] = t[b, a]
    return committed, bonus


def verify(logits: np.ndarray, draft: np.ndarray) -> dict:
    """Greedy verification of a block: target argmax, A, committed, bonus."""
    t = target_argmax(logits)
    A = accepted_length(t, draft)
    committed, bonus = commit(t, draft, A)
    return {"target_argmax": t, "accept_len": A, "committed": committed, "bonus": bonus}


# ---------------------------------------------------------------------------
# Rejected-trajectory conditioning (Eq. 3-8, Algorithm 1 carry/reset steps)
# ---------------------------------------------------------------------------


def carried_rows(A: np.ndarray, K: int) -> np.ndarray:
    """n_b = number of aligned positions that receive a signal next round.

    Eq. 4 carries h^D_{t, r_t+j} for 1 <= j <= B - r_t (paper indices), i.e.
    K - (A + 1) rows; Algorithm 1 resets the carry when A_t >= K - 1 (full
    acceptance, or rejection at the last slot).  Both give max(0, K-1-A).
    """
    return np.maximum(0, K - 1 - np.asarray(A, dtype=np.int64))


def align(hD: np.ndarray, hT: np.ndarray, A: np.ndarray):
    """Aligned draft trajectory m (Eq. 4) and target states u (Eq. 5).

    With 0-based slots, row j < n_b of the next block receives
    m[b, j] = hD[b, A_b + 1 + j]  (the states strictly after the first
    rejected slot, shifted to the start of the block, order preserved) and
    u[b, j] = hT[b, A_b + j]  (the target state whose logits score the same
    slot A_b + 1 + j).  Rows j >= n_b are zero.
    """
    hD = np.asarray(hD, dtype=np.float64)
    hT = np.asarray(hT, dtype=np.float64)
    B, K, d = hD.shape
    n = carried_rows(A, K)
    m = np.zeros((B, K, d), dtype=np.float64)
    u = np.zeros((B, K, d), dtype=np.float64)
    for b in range(B):
        a = int(A[b])
        for j in range(int(n[b])):
            m[b, j] = hD[b, a + 1 + j]
            u[b, j] = hT[b, a + j]
    return m, u


def correct(m: np.ndarray, u: np.ndarray, Wc: np.ndarray, beta: float, round_r_bf16: bool):
    """Target-aware correction: c = W_c [m; u] (Eq. 6), r = m + beta c (Eq. 7).

    ``[m; u]`` is the concatenation along the hidden dimension (length 2d) and
    W_c is [d, 2d].  When ``round_r_bf16`` the corrected signal is rounded to
    bfloat16, the precision in which the GPU path stores it between the two
    projections; otherwise it stays float64.
    """
    x = np.concatenate([m, u], axis=-1)  # [B, K, 2d]
    c = x @ np.asarray(Wc, dtype=np.float64).T  # [B, K, d]
    r = m + float(beta) * c
    return round_to_bf16(r) if round_r_bf16 else r


def sigmoid(z: np.ndarray) -> np.ndarray:
    """Element-wise logistic function 1 / (1 + exp(-z)), evaluated without overflow."""
    z = np.asarray(z, dtype=np.float64)
    out = np.empty_like(z)
    pos = z >= 0
    out[pos] = 1.0 / (1.0 + np.exp(-z[pos]))
    ez = np.exp(z[~pos])
    out[~pos] = ez / (1.0 + ez)
    return out


def gate_fuse(e: np.ndarray, r: np.ndarray, n: np.ndarray, Wv: np.ndarray, Wg: np.ndarray):
    """Gated residual conditioning (Eq. 8), float64.

    For conditioned rows j < n_b:  e~ = e + (W_v r) * sigmoid(W_g [e; r]),
    with a vector-valued gate; every other position keeps e exactly
    (Sec. 4.1: positions without an aligned signal keep their inputs).
    ``e`` is [B, K, d] (broadcast a single mask embedding before calling).
    """
    e = np.asarray(e, dtype=np.float64)
    r = np.asarray(r, dtype=np.float64)
    B, K, d = e.shape
    v = r @ np.asarray(Wv, dtype=np.float64).T
    g = np.concatenate([e, r], axis=-1) @ np.asarray(Wg, dtype=np.float64).T
    fused = e + v * sigmoid(g)
    rows = np.arange(K)[None, :] < np.asarray(n)[:, None]  # [B, K]
    return np.where(rows[..., None], fused, e)


VARIANTS = ("corrected", "raw", "overwrite", "none")


def condition(e_full, m, u, n, Wc, Wv, Wg, beta, variant: str, round_r_bf16: bool):
    """How the aligned signal enters the next block; returns (r, e~).

    The component ablation (Sec. "Component Ablation", Table 3; Appendix
    "Ablation Settings") compares variants that build the same aligned
    signal m (Eq. 4) and differ only in how it is used:

    * ``corrected``: the method, r = m + beta W_c [m; u] (Eq. 6-7), then the
      gated fusion of Eq. 8;
    * ``raw``: the gated fusion of Eq. 8 without correction, r = m;
    * ``overwrite``: the aligned states replace the mask inputs, e~_j = m_j;
    * ``none``: no conditioning (the DFlash row of Table 3), e~ = e.

    In every variant positions j >= n_b keep e.  r is None where a variant
    has none.
    """
    if variant == "corrected":
        r = correct(m, u, Wc, beta, round_r_bf16)
        return r, gate_fuse(e_full, r, n, Wv, Wg)
    if variant == "raw":
        return m, gate_fuse(e_full, m, n, Wv, Wg)
    K = m.shape[1]
    rows = np.arange(K)[None, :] < np.asarray(n)[:, None]  # [B, K]
    if variant == "overwrite":
        return None, np.where(rows[..., None], m, e_full)
    if variant == "none":
        return None, np.array(e_full, dtype=np.float64, copy=True)
    raise ValueError(f"unknown variant {variant!r}")


def retrace_round(logits, draft, hD, hT, e, Wc, Wv, Wg, beta, dtype: str, variant: str = "corrected") -> dict:
    """One round: verify, then condition the next block (Algorithm 1).

    ``dtype`` is "bf16" or "f32", the precision of the GPU path being checked;
    it decides only whether r and the output are rounded to bfloat16.
    ``variant`` is one of ``VARIANTS`` (see :func:`condition`).
    Returns the verification outputs plus ``n``, ``r`` and ``e_tilde``
    (float64) and, for bf16, ``e_tilde_rounded``.
    """
    out = verify(logits, draft)
    A = out["accept_len"]
    K = np.asarray(draft).shape[1]
    n = carried_rows(A, K)
    m, u = align(hD, hT, A)
    e_full = np.broadcast_to(np.asarray(e, dtype=np.float64), np.asarray(hD).shape)
    r, e_tilde = condition(e_full, m, u, n, Wc, Wv, Wg, beta, variant, round_r_bf16=(dtype == "bf16"))
    out.update({"n": n, "r": r, "e_tilde": e_tilde})
    if dtype == "bf16":
        out["e_tilde_rounded"] = round_to_bf16(e_tilde)
    return out


def conditioned_rows(rows, A, hD, hT, e, Wc, Wv, Wg, beta, dtype: str) -> np.ndarray:
    """e~ for a list of (b, j) positions only, by the same equations.

    Used to check full-size workloads on a sample of rows: each row of Eq. 4-8
    depends only on its own sequence's A_b, its own two hidden states and the
    weights, so it can be evaluated alone.  Returns float64 [len(rows), d]
    (rounded to bf16 values when dtype == "bf16").
    """
    Wc = np.asarray(Wc, dtype=np.float64)
    Wv = np.asarray(Wv, dtype=np.float64)
    Wg = np.asarray(Wg, dtype=np.float64)
    K = np.asarray(hD).shape[1]
    out = []
    for b, j in rows:
        a = int(A[b])
        n_b = max(0, K - 1 - a)
        e_bj = np.asarray(e[b, j] if np.ndim(e) == 3 else e, dtype=np.float64)
        if j >= n_b:
            out.append(e_bj.copy())
            continue
        m = np.asarray(hD[b, a + 1 + j], dtype=np.float64)
        u = np.asarray(hT[b, a + j], dtype=np.float64)
        r = m + float(beta) * (Wc @ np.concatenate([m, u]))
        if dtype == "bf16":
            r = round_to_bf16(r)
        v = Wv @ r
        g = Wg @ np.concatenate([e_bj, r])
        out.append(e_bj + v * sigmoid(g))
    res = np.stack(out) if out else np.zeros((0, np.asarray(hD).shape[2]))
    return round_to_bf16(res) if dtype == "bf16" else res


# ---------------------------------------------------------------------------
# Low-rank realisation of the conditioning (Appendix "Concurrent-Serving
# Experiment"): rank-64 rejected-suffix latents, a rank-32 target-aware
# correction, and input-side latent residual fusion, for one round.
# ---------------------------------------------------------------------------

LOWRANK_LATENT = 64
LOWRANK_CORRECTION = 32


def lowrank_condition(e_full, m, u, n, P, Bc, Ac, Wv, Wg, beta, round_bf16: bool):
    """The conditioning path with low-rank factors; returns (z, rho, e~).

    The appendix names the parts without equations; this is the reading used
    here, the method's Eq. 6-8 with every d-wide signal replaced by a rank-64
    latent and the correction factored through rank 32:

    * latent of the rejected drafter state:  z = P m            (P: [64, d])
    * rank-32 target-aware correction:      rho = z + beta A_c (B_c [z; u])
                                             (B_c: [32, 64 + d], A_c: [64, 32])
    * input-side latent residual fusion:    e~ = e + (W_v rho) * sigmoid(W_g [e; rho])
                                             (W_v: [d, 64], W_g: [d, d + 64])

    Rows j >= n_b keep e.  With ``round_bf16`` the latent z and rho are
    rounded to bfloat16 where the GPU stores them (z as the carried latent,
    rho as the input of the up-projections).
    """
    P = np.asarray(P, dtype=np.float64)
    Bc = np.asarray(Bc, dtype=np.float64)
    Ac = np.asarray(Ac, dtype=np.float64)
    z = np.asarray(m, dtype=np.float64) @ P.T  # [B, K, 64]
    if round_bf16:
        z = round_to_bf16(z)
    t = np.concatenate([z, np.asarray(u, dtype=np.float64)], axis=-1) @ Bc.T  # [B, K, 32]
    rho = z + float(beta) * (t @ Ac.T)
    if round_bf16:
        rho = round_to_bf16(rho)
    e_full = np.asarray(e_full, dtype=np.float64)
    v = rho @ np.asarray(Wv, dtype=np.float64).T
    g = np.concatenate([e_full, rho], axis=-1) @ np.asarray(Wg, dtype=np.float64).T
    fused = e_full + v * sigmoid(g)
    K = e_full.shape[1]
    rows = np.arange(K)[None, :] < np.asarray(n)[:, None]
    return z, rho, np.where(rows[..., None], fused, e_full)


def retrace_round_lowrank(logits, draft, hD, hT, e, P, Bc, Ac, Wv, Wg, beta, dtype: str) -> dict:
    """One round with the low-rank conditioning path (see lowrank_condition)."""
    out = verify(logits, draft)
    A = out["accept_len"]
    K = np.asarray(draft).shape[1]
    n = carried_rows(A, K)
    m, u = align(hD, hT, A)
    e_full = np.broadcast_to(np.asarray(e, dtype=np.float64), np.asarray(hD).shape)
    z, rho, e_tilde = lowrank_condition(e_full, m, u, n, P, Bc, Ac, Wv, Wg, beta, round_bf16=(dtype == "bf16"))
    out.update({"n": n, "z": z, "rho": rho, "e_tilde": e_tilde})
    if dtype == "bf16":
        out["e_tilde_rounded"] = round_to_bf16(e_tilde)
    return out


# ---------------------------------------------------------------------------
# Stochastic verification at temperature T (Appendix "Evaluation Protocol":
# T = 1 with top_p = 0.95 and top_k = 20).  The paper keeps the underlying
# speculative-decoding verification and does not state it; the reading used
# here is standard speculative sampling on the filtered distributions, with
# the random numbers passed in as inputs.
# ---------------------------------------------------------------------------


def filtered_distribution(logits_row, T: float, top_k: int, top_p: float):
    """Tokens and probabilities of the sampling distribution of one row.

    softmax(logits / T), restricted to the top_k largest logits (the lowest
    index first among equal values), renormalised, then restricted to the
    shortest prefix of those tokens, in that order, whose probability sums to
    at least top_p, and renormalised again.  Returns (tokens, probs) in that
    order (descending probability).
    """
    x = np.asarray(logits_row, dtype=np.float64)
    idx = np.arange(x.shape[0])
    order = np.lexsort((idx, -x))[:top_k]  # descending value, ascending index
    w = np.exp((x[order] - x[order[0]]) / float(T))
    p = w / w.sum()
    keep = int(np.searchsorted(np.cumsum(p), top_p, side="left")) + 1  # first prefix reaching top_p
    keep = min(keep, len(order))
    w = w[:keep]
    return order[:keep], w / w.sum()


def _prob_of(tokens, probs, y):
    hit = np.flatnonzero(tokens == y)
    return float(probs[hit[0]]) if hit.size else 0.0


def _sample(tokens, probs, u: float) -> int:
    """Inverse-CDF draw in the given token order: the first token whose
    cumulative probability exceeds u (u in [0, 1))."""
    c = np.cumsum(probs)
    j = int(np.searchsorted(c, u * c[-1], side="right"))
    return int(tokens[min(j, len(tokens) - 1)])


def verify_sampled(target_logits, draft_logits, draft, uniforms, T: float, top_k: int, top_p: float) -> dict:
    """Speculative sampling of one block per sequence.

    With p_i and q_i the filtered target and draft distributions of slot i,
    draft token x_i is accepted iff u_i q_i(x_i) < p_i(x_i), i.e. with
    probability min(1, p_i(x_i) / q_i(x_i)); verification stops at the first
    rejection A.  The token appended after the accepted prefix is drawn with
    u_K: from the residual max(0, p_A - q_A) (renormalised; from p_A if it is
    zero everywhere) when A < K, from p_K when every draft was accepted.
    A draft token outside [0, V) is rejected.
    """
    tl = np.asarray(target_logits)
    dl = np.asarray(draft_logits)
    draft = np.asarray(draft)
    u = np.asarray(uniforms, dtype=np.float64)
    B, K = draft.shape
    V = tl.shape[2]
    A = np.full(B, K, dtype=np.int64)
    committed = np.full((B, K + 1), -1, dtype=np.int64)
    bonus = np.empty(B, dtype=np.int64)
    for b in range(B):
        a = K
        for i in range(K):
            x = int(draft[b, i])
            pt, pp = filtered_distribution(tl[b, i], T, top_k, top_p)
            qt, qp = filtered_distribution(dl[b, i], T, top_k, top_p)
            px = _prob_of(pt, pp, x) if 0 <= x < V else 0.0
            qx = _prob_of(qt, qp, x) if 0 <= x < V else 0.0
            if not (0 <= x < V and u[b, i] * qx < px):
                a = i
                break
        pt, pp = filtered_distribution(tl[b, a], T, top_k, top_p)
        if a < K:
            qt, qp = filtered_distribution(dl[b, a], T, top_k, top_p)
            res = np.array([max(0.0, pp[j] - _prob_of(qt, qp, int(pt[j]))) for j in range(len(pt))])
            y = _sample(pt, res, u[b, K]) if res.sum() > 0 else _sample(pt, pp, u[b, K])
        else:
            y = _sample(pt, pp, u[b, K])
        A[b] = a
        committed[b, :a] = draft[b, :a]
        committed[b, a] = y
        bonus[b] = y
    return {"accept_len": A, "committed": committed, "bonus": bonus}
