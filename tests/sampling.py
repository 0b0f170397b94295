"""Helpers of the sampled-verification parity tests.

Floating point decides the accept tests, the top-p cut and the draws; the GPU
computes them in fp32 and the oracle in float64.  The uniforms are inputs, so
the tests move any uniform that lies within a small margin of its decision
boundary (measure-zero cases) and mark the sequences whose top-p cut itself is
that close; those sequences are checked for validity instead of equality.
"""

import numpy as np

import oracle

MARGIN = 2e-3


def _dist(row, T, k, p):
    return oracle.filtered_distribution(row, T, k, p)


def _prob(dist, y):
    toks, ps = dist
    hit = np.flatnonzero(toks == y)
    return float(ps[hit[0]]) if hit.size else 0.0


def _cut_is_close(row, T, k, p):
    x = np.asarray(row, dtype=np.float64)
    order = np.lexsort((np.arange(x.size), -x))[:k]
    w = np.exp((x[order] - x[order[0]]) / T)
    c = np.cumsum(w / w.sum())[:-1]  # the last entry is kept whenever every earlier one is
    return bool(np.any(np.abs(c - p) < 1e-5 * max(p, 1e-30)))


def conditioned_uniforms(tl, dl, draft, u, T, k, p):
    """Moves uniforms away from the decision boundaries of the oracle's run;
    returns (uniforms, ambiguous sequences)."""
    B, K = draft.shape
    u = u.copy()
    ambiguous = set()
    for b in range(B):
        a = K
        for i in range(K):
            if _cut_is_close(tl[b, i], T, k, p) or _cut_is_close(dl[b, i], T, k, p):
                ambiguous.add(b)
            x = int(draft[b, i])
            px, qx = _prob(_dist(tl[b, i], T, k, p), x), _prob(_dist(dl[b, i], T, k, p), x)
            if qx > 0 and abs(u[b, i] * qx - px) < MARGIN * max(px, qx):
                u[b, i] = min(max(px / qx + (3 * MARGIN if u[b, i] * qx >= px else -3 * MARGIN), 0.0), 0.999)
            if not u[b, i] * qx < px:
                a = i
                break
        if _cut_is_close(tl[b, a], T, k, p):
            ambiguous.add(b)
        pt, pp = _dist(tl[b, a], T, k, p)
        if a < K:
            qd = _dist(dl[b, a], T, k, p)
            w = np.array([max(0.0, pp[j] - _prob(qd, int(pt[j]))) for j in range(len(pt))])
            if w.sum() <= 0:
                w = pp
        else:
            w = pp
        steps = np.cumsum(w) / w.sum()
        while np.any(np.abs(steps - u[b, K]) < MARGIN):
            u[b, K] = (u[b, K] + 0.37 * MARGIN * 7) % 1.0
    return u, ambiguous
