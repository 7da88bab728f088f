"""Pure-Python brute force for tiny inputs (test infrastructure only).

Each function builds the paper's full intermediate matrices explicitly with
Python lists and ``math`` (no numpy), so the C oracle can be checked against a
second, independent restatement on inputs small enough to enumerate
(N_t <= 8, N_v <= 16, L <= 40).
"""
from __future__ import annotations

import math


def _dot(a, b):
    return sum(x * y for x, y in zip(a, b))


def _softmax(xs):
    m = max(xs)
    ex = [math.exp(x - m) for x in xs]
    z = sum(ex)
    return [e / z for e in ex]


def crit_text(E):
    """Sec. 4.2 with the full N_t x N_t softmax matrix written out."""
    n = len(E)
    G = [[_dot(E[i], E[j]) for j in range(n)] for i in range(n)]
    R = [_softmax(G[i]) for i in range(n)]
    r = [sum(R[i][j] for i in range(n)) / n for j in range(n)]
    mean = sum(r) / n
    T = [j for j in range(n) if r[j] > mean]
    if not T:
        T = list(range(n))
    return r, T


def _cos(a, b):
    na, nb = math.sqrt(_dot(a, a)), math.sqrt(_dot(b, b))
    if na == 0.0 or nb == 0.0:
        return 0.0
    return _dot(a, b) / (na * nb)


def relevance(Et, T, Ev):
    """Sec. 4.3: explicit |T| x N_v cosine matrix, de-meaned rows, column max."""
    M = [[_cos(Et[i], v) for v in Ev] for i in T]
    Mh = [[x - sum(row) / len(row) for x in row] for row in M]
    return [max(Mh[a][j] for a in range(len(T))) for j in range(len(Ev))]


def topk(s, k):
    order = sorted(range(len(s)), key=lambda i: (-s[i], i))
    return sorted(order[:k])


def merge(Ev, keep):
    """Sec. 4.3 merge reading: full pruned x kept cosine matrix, row argmax."""
    kept = set(keep)
    assign = []
    for j, e in enumerate(Ev):
        if j in kept:
            assign.append(keep.index(j))
            continue
        cs = [_cos(e, Ev[k]) for k in keep]
        best = 0
        for a in range(1, len(cs)):
            if cs[a] > cs[best]:
                best = a
        assign.append(best)
    d = len(Ev[0])
    merged = []
    for a in range(len(keep)):
        members = [Ev[j] for j in range(len(Ev)) if assign[j] == a]
        merged.append([sum(m[e] for m in members) / len(members) for e in range(d)])
    return assign, merged


def attention_matrix(Q, K, h, group):
    """Full L x L causal attention matrix of query head h (Q[t][h], K[t][g])."""
    L = len(Q)
    dh = len(Q[0][0])
    g = h // group
    A = []
    for t in range(L):
        logits = [(_dot(Q[t][h], K[k][g]) / math.sqrt(dh)) if k <= t else -math.inf
                  for k in range(L)]
        m = max(x for x in logits if x != -math.inf)
        ex = [math.exp(x - m) if x != -math.inf else 0.0 for x in logits]
        z = sum(ex)
        A.append([e / z for e in ex])
    return A


def head_scores(Q, K, heads, rows, vis_start, nv):
    """Sec. 4.4: slice A^cross out of the full attention matrices, average."""
    Hq, Hkv = len(Q[0]), len(K[0])
    group = Hq // Hkv
    mats = {h: attention_matrix(Q, K, h, group) for h in heads}
    v = [0.0] * nv
    for t in rows:
        for i in range(nv):
            S = sum(mats[h][t][vis_start + i] for h in heads) / len(heads)
            v[i] += S / len(rows)
    return v


def head_confidence(Q, K, rows, vis_start, nv):
    Hq, Hkv = len(Q[0]), len(K[0])
    group = Hq // Hkv
    C = []
    for h in range(Hq):
        A = attention_matrix(Q, K, h, group)
        c = 0.0
        for t in rows:
            xs = A[t][vis_start:vis_start + nv]
            mu = sum(xs) / nv
            c += sum((x - mu) ** 2 for x in xs) / nv
        C.append(c)
    return C
