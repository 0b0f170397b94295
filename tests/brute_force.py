"""Pure-Python brute force for tiny ReTrace rounds (pins the oracle).

Independent of ``oracle/``: plain lists and ``math`` only, each step computed
by a different route than the oracle takes -- the argmax by a full stable sort,
the accepted length by trying every candidate length, the projections as
explicit sums over separately indexed halves of the weight matrices.
"""

import math


def argmax_by_sort(row):
    """Index of the maximum, lowest index on ties (-0.0 == +0.0): stable sort by value, descending."""
    order = sorted(range(len(row)), key=lambda v: -row[v])  # sorted() is stable
    return order[0]


def accept_len_by_search(t, draft):
    """Largest a such that t[i] == draft[i] for every i < a."""
    K = len(draft)
    best = 0
    for a in range(K + 1):
        if all(t[i] == draft[i] for i in range(a)):
            best = a
    return best


def round_brute(logits, draft, hD, hT, e, Wc, Wv, Wg, beta, rnd=None):
    """One sequence's round.  ``rnd`` (optional) rounds r before the gate.

    logits [K+1][V], draft [K], hD/hT [K][d], e [K][d], Wc [d][2d], Wv [d][d], Wg [d][2d].
    """
    K = len(draft)
    d = len(Wv)
    t = [argmax_by_sort(logits[i]) for i in range(K + 1)]
    A = accept_len_by_search(t, draft)
    committed = [draft[i] for i in range(A)] + [t[A]]
    n = 0
    for j in range(K):
        # slot of the next block that still has a rejected state after the
        # first rejected slot: A + 1 + j must be a valid draft slot
        if A + 1 + j <= K - 1:
            n += 1
    out = []
    for j in range(K):
        if j >= n:
            out.append(list(e[j]))
            continue
        m = hD[A + 1 + j]
        u = hT[A + j]
        r = []
        for i in range(d):
            c = sum(Wc[i][k] * m[k] for k in range(d)) + sum(Wc[i][d + k] * u[k] for k in range(d))
            r.append(m[i] + beta * c)
        if rnd is not None:
            r = rnd(r)
        row = []
        for i in range(d):
            v = sum(Wv[i][k] * r[k] for k in range(d))
            g = sum(Wg[i][k] * e[j][k] for k in range(d)) + sum(Wg[i][d + k] * r[k] for k in range(d))
            row.append(e[j][i] + v * (1.0 / (1.0 + math.exp(-g))))
        out.append(row)
    return {"t": t, "A": A, "committed": committed, "bonus": t[A], "n": n, "e_tilde": out}


def lowrank_brute(logits, draft, hD, hT, e, P, Bc, Ac, Wv, Wg, beta, rnd=None):
    """One sequence's round with the low-rank conditioning, by explicit sums.

    P [L][d], Bc [C][L + d] (columns 0..L-1 act on the latent), Ac [L][C],
    Wv [d][L], Wg [d][d + L] (columns 0..d-1 act on e).  ``rnd`` (optional)
    rounds the latent and the corrected latent.
    """
    K = len(draft)
    d = len(Wv)
    L = len(P)
    C = len(Bc)
    t = [argmax_by_sort(logits[i]) for i in range(K + 1)]
    A = accept_len_by_search(t, draft)
    n = sum(1 for j in range(K) if A + 1 + j <= K - 1)
    out = []
    for j in range(K):
        if j >= n:
            out.append(list(e[j]))
            continue
        m = hD[A + 1 + j]
        u = hT[A + j]
        z = [sum(P[i][k] * m[k] for k in range(d)) for i in range(L)]
        if rnd is not None:
            z = rnd(z)
        tc = [sum(Bc[c][i] * z[i] for i in range(L)) + sum(Bc[c][L + k] * u[k] for k in range(d)) for c in range(C)]
        rho = [z[i] + beta * sum(Ac[i][c] * tc[c] for c in range(C)) for i in range(L)]
        if rnd is not None:
            rho = rnd(rho)
        row = []
        for f in range(d):
            v = sum(Wv[f][i] * rho[i] for i in range(L))
            g = sum(Wg[f][k] * e[j][k] for k in range(d)) + sum(Wg[f][d + i] * rho[i] for i in range(L))
            row.append(e[j][f] + v * (1.0 / (1.0 + math.exp(-g))))
        out.append(row)
    return {"t": t, "A": A, "n": n, "e_tilde": out}
