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


def filtered_brute(row, T, top_k, top_p):
    """Sampling distribution of one row by explicit loops: a full sort by
    (value descending, index ascending), the first top_k, softmax at T over
    them, the shortest prefix reaching top_p, renormalised."""
    order = sorted(range(len(row)), key=lambda v: (-row[v], v))[:top_k]
    w = [math.exp((row[v] - row[order[0]]) / T) for v in order]
    total = sum(w)
    acc, keep = 0.0, len(order)
    for j in range(len(order)):
        acc += w[j] / total
        if acc >= top_p:
            keep = j + 1
            break
    z = sum(w[:keep])
    return order[:keep], [x / z for x in w[:keep]]


def sampled_brute(tlog, dlog, draft, u, T, top_k, top_p):
    """One sequence of speculative sampling (accept iff u_i q(x) < p(x);
    residual max(0, p - q) at the first rejection, else p at slot K;
    inverse CDF in the filtered order)."""
    K = len(draft)
    V = len(tlog[0])

    def prob(dist, y):
        toks, ps = dist
        return ps[toks.index(y)] if y in toks else 0.0

    def draw(toks, ws, r):
        total = sum(ws)
        acc = 0.0
        for t, w in zip(toks, ws):
            acc += w
            if acc > r * total:
                return t
        return toks[-1]

    a = K
    for i in range(K):
        x = draft[i]
        ok = False
        if 0 <= x < V:
            ok = u[i] * prob(filtered_brute(dlog[i], T, top_k, top_p), x) < prob(filtered_brute(tlog[i], T, top_k, top_p), x)
        if not ok:
            a = i
            break
    pd = filtered_brute(tlog[a], T, top_k, top_p)
    if a < K:
        qd = filtered_brute(dlog[a], T, top_k, top_p)
        res = [max(0.0, pd[1][j] - prob(qd, pd[0][j])) for j in range(len(pd[0]))]
        y = draw(pd[0], res, u[K]) if sum(res) > 0 else draw(pd[0], pd[1], u[K])
    else:
        y = draw(pd[0], pd[1], u[K])
    return {"A": a, "committed": list(draft[:a]) + [y]}
