"""Brute-force statement of one MoECa layer step for tiny cases (T <= 8, E <= 4).

Pure Python loops over float64 scalars, written separately from the oracle:
every expert's FFN output is computed densely for every token (Eq. 5), the
routing is a full sort of all experts, matching is a linear search of the cache
(Sec. 4.2), the entropy is summed term by term (Eq. 11) and the combine is the
literal Eq. 8.  Decisions compare float32-rounded values, as the oracle does.
"""
from __future__ import annotations

import math

import numpy as np


def _f32(x: float) -> float:
    return float(np.float32(x))


def _gelu(z: float, form: str) -> float:
    if form == "tanh":
        return 0.5 * z * (1.0 + math.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z * z * z)))
    return 0.5 * z * (1.0 + math.erf(z / math.sqrt(2.0)))


def _ffn(u, w1, w2, form):
    F, D = len(w1), len(u)
    mid = [_gelu(sum(float(w1[f][d]) * u[d] for d in range(D)), form) for f in range(F)]
    return [sum(float(w2[d][f]) * mid[f] for f in range(F)) for d in range(D)]


def layer_step(state: dict, x, wts: dict, prm: dict, refresh: bool):
    """state: dict of python lists {cache_e, cache_w, cache_norm, cache_h, shared_h, C}.

    C is indexed C[e][i] as in Eq. 10.  Returns (out, new_state, decisions).
    """
    T, D = len(x), len(x[0])
    E = len(wts["w_gate"])
    k = prm["top_k"]
    u = [[float(v) for v in row] for row in x]
    # Dense: every expert on every token.
    dense = [[_ffn(u[i], wts["w1"][e], wts["w2"][e], prm["gelu"]) for e in range(E)] for i in range(T)]
    # Routing by a full sort of (float32 logit desc, expert id asc).
    e_cur, w_cur = [], []
    for i in range(T):
        z = []
        for e in range(E):
            v = sum(float(wts["w_gate"][e][d]) * u[i][d] for d in range(D))
            if wts.get("b_gate") is not None:
                v += float(wts["b_gate"][e])
            z.append(v)
        ranked = sorted(range(E), key=lambda e: (-_f32(z[e]), e))
        m = max(z)
        ex = [math.exp(v - m) for v in z]
        tot = sum(ex)
        probs = [v / tot for v in ex]
        pick = ranked[:k]
        w = [probs[e] for e in pick]
        if prm["renorm_topk"]:
            sw = sum(w)
            w = [v / sw for v in w]
        e_cur.append(pick)
        w_cur.append(w)
    # EMA statistic (Eq. 10).
    beta = prm["beta"]
    C = [[beta * state["C"][e][i] + (1.0 - beta) * (1.0 if e in e_cur[i] else 0.0) for i in range(T)]
         for e in range(E)]
    # Entropy, normalisation and threshold (Eq. 11, Eq. 12).
    Hs = []
    for e in range(E):
        S = sum(C[e])
        if S <= 0.0:
            Hs.append(None)
            continue
        H = 0.0
        for i in range(T):
            P = C[e][i] / S
            if P > 0.0:
                H -= P * math.log(P)
        Hs.append(H)
    Hbar = []
    if prm["entropy_norm"] == "log_t":
        for H in Hs:
            Hbar.append(0.5 if (H is None or T <= 1) else min(1.0, max(0.0, H / math.log(T))))
    else:
        live = [H for H in Hs if H is not None]
        lo, hi = (min(live), max(live)) if live else (0.0, 0.0)
        for H in Hs:
            Hbar.append(0.5 if (H is None or hi <= lo) else (H - lo) / (hi - lo))
    tau = [prm["tau0"] * (1.0 + prm["alpha"] * (2.0 * hb - 1.0)) for hb in Hbar]
    # Decisions.
    rec = [[True] * k for _ in range(T)]
    slot = [list(range(k)) for _ in range(T)]
    if not refresh:
        for i in range(T):
            norms = state["cache_norm"][i]
            tot = sum(norms)
            taken = []
            for p in range(k):
                q_hit = None
                for q in range(k):
                    if state["cache_e"][i][q] == e_cur[i][p]:
                        q_hit = q
                        break
                if q_hit is None:
                    taken.append(None)
                    continue
                taken.append(q_hit)
                delta = abs(w_cur[i][p] - state["cache_w"][i][q_hit])
                o = norms[q_hit] / tot if tot > 0.0 else 0.0
                terms = prm.get("score_terms", 7)
                s = 0.0
                if terms & 1:
                    s += w_cur[i][p]
                if terms & 2:
                    s += prm["lambda1"] * delta
                if terms & 4:
                    s += prm["lambda2"] * o
                rec[i][p] = _f32(s) > _f32(tau[e_cur[i][p]])
            if prm.get("granularity", "branch") == "token" and True in rec[i]:
                rec[i] = [True] * k
            free = [q for q in range(k) if q not in taken]
            for p in range(k):
                if taken[p] is not None:
                    slot[i][p] = taken[p]
                else:
                    slot[i][p] = free.pop(0)
    # Cache update, shared experts, combine (Eq. 8) and norms.
    ce = [list(r) for r in state["cache_e"]]
    cw = [list(r) for r in state["cache_w"]]
    ch = [[list(h) for h in r] for r in state["cache_h"]]
    sh = None if state["shared_h"] is None else [list(r) for r in state["shared_h"]]
    for i in range(T):
        for p in range(k):
            q = slot[i][p]
            if rec[i][p]:
                ch[i][q] = list(dense[i][e_cur[i][p]])
                ce[i][q] = e_cur[i][p]
                cw[i][q] = w_cur[i][p]
            elif prm["reused_meta_policy"] == "overwrite":
                cw[i][q] = w_cur[i][p]
    if sh is not None:
        for i in range(T):
            if refresh or prm["shared_policy"] == "always" or any(rec[i]):
                sh[i] = [0.0] * D
                for s in range(len(wts["ws1"])):
                    hs = _ffn(u[i], wts["ws1"][s], wts["ws2"][s], prm["gelu"])
                    sh[i] = [a + b for a, b in zip(sh[i], hs)]
    out = []
    for i in range(T):
        y = [0.0] * D
        for p in range(k):
            h = ch[i][slot[i][p]]
            for d in range(D):
                y[d] += w_cur[i][p] * h[d]
        if sh is not None:
            for d in range(D):
                y[d] += sh[i][d]
        out.append([u[i][d] + y[d] for d in range(D)])
    cn = [[math.sqrt(sum(v * v for v in ch[i][q])) for q in range(k)] for i in range(T)]
    new = dict(cache_e=ce, cache_w=cw, cache_norm=cn, cache_h=ch, shared_h=sh, C=C)
    dec = dict(e=e_cur, w=w_cur, recompute=rec, slot=slot, tau=tau)
    return out, new, dec


def empty_state(T, D, E, k, n_shared):
    return dict(cache_e=[[-1] * k for _ in range(T)], cache_w=[[0.0] * k for _ in range(T)],
                cache_norm=[[0.0] * k for _ in range(T)],
                cache_h=[[[0.0] * D for _ in range(k)] for _ in range(T)],
                shared_h=[[0.0] * D for _ in range(T)] if n_shared else None,
                C=[[0.0] * T for _ in range(E)])
