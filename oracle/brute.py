"""Pure-Python brute force for tiny CommitKV problems — TEST INFRASTRUCTURE.

Written separately from ``commitkv_oracle.c`` (no shared code), with
nested lists and ``math`` only, so that a mistake in one of the two is
caught by the other.  Every page subset of a problem with a handful of
pages is deleted explicitly (Section 3.2, Eq. 6-7 and Eq. 11).

Problem layout: K[l][kvh][i][c], V likewise, Q[l][h][w][c], pos[i],
qpos[w], pages = list of (start, length).
"""
from __future__ import annotations

import itertools
import math

INF = float("inf")


def _softmax_out(scores, values, keep):
    idx = [i for i in range(len(scores)) if keep[i]]
    if not idx:
        return None
    m = max(scores[i] for i in idx)
    w = {i: math.exp(scores[i] - m) for i in idx}
    tot = math.fsum(w.values())
    d = len(values[0])
    return [math.fsum(w[i] * values[i][c] for i in idx) / tot for c in range(d)]


def row_effect(q, keys, values, pos, qp, deleted, scale):
    """Relative change of one head's output at one query when the token set
    `deleted` is removed (degenerate rules: nothing visible deleted -> 0,
    everything visible deleted -> inf, zero output -> 0 or inf)."""
    S = len(keys)
    vis = [pos[i] <= qp for i in range(S)]
    scores = [scale * math.fsum(a * b for a, b in zip(q, keys[i])) for i in range(S)]
    n_vis = sum(vis)
    n_del = sum(1 for i in range(S) if vis[i] and i in deleted)
    if n_del == 0:
        return 0.0
    if n_del == n_vis:
        return INF
    o = _softmax_out(scores, values, vis)
    o2 = _softmax_out(scores, values, [vis[i] and i not in deleted for i in range(S)])
    num = math.sqrt(math.fsum((a - b) ** 2 for a, b in zip(o, o2)))
    den = math.sqrt(math.fsum(a * a for a in o))
    if den == 0.0:
        return 0.0 if num == 0.0 else INF
    return num / den


def set_effect(prob, token_set, layers=None):
    K, V, Q, pos, qpos = prob["K"], prob["V"], prob["Q"], prob["pos"], prob["qpos"]
    M, H, Hq = len(K), len(K[0]), len(Q[0])
    d = len(K[0][0][0])
    scale = prob.get("scale") or 1.0 / math.sqrt(d)
    g = Hq // H
    R = 0.0
    for l in range(M):
        if layers is not None and not layers[l]:
            continue
        for h in range(Hq):
            for w, qp in enumerate(qpos):
                r = row_effect(Q[l][h][w], K[l][h // g], V[l][h // g], pos, qp, token_set, scale)
                R = max(R, r)
    return R


def page_tokens(prob, pages_subset):
    toks = set()
    for E in pages_subset:
        b, n = prob["pages"][E]
        toks.update(range(b, b + n))
    return toks


def all_subset_effects(prob, layers=None):
    """{frozenset(pages): R(A)} for every subset A of the pages."""
    P = len(prob["pages"])
    out = {}
    for r in range(P + 1):
        for A in itertools.combinations(range(P), r):
            out[frozenset(A)] = set_effect(prob, page_tokens(prob, A), layers)
    return out


def greedy_from_table(table, cand, tau):
    """Greedy joint test re-derived from a table of set effects."""
    D = frozenset()
    steps = []
    for E in cand:
        R = table[D | {E}]
        steps.append(R)
        if R <= tau:
            D = D | {E}
    return D, steps
