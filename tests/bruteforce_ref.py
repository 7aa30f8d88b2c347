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


def layer_step(state: dict, x, wts: dict, prm: dict, refresh: bool, ffn_input=None, resid=None, gate=None):
    """state: dict of python lists {cache_e, cache_w, cache_norm, cache_h, shared_h, C}.

    C is indexed C[e][i] as in Eq. 10.  Returns (out, new_state, decisions).
    x is the router input.  An AdaLN block passes ``ffn_input(rec)``, which
    returns the FFN rows once the recompute sets are known (the sync rule
    recomputes attention in between), and the output resid + gate * y.
    """
    T, D = len(x), len(x[0])
    E = len(wts["w_gate"])
    k = prm["top_k"]
    u = [[float(v) for v in row] for row in x]
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
    # Dense: every expert on every token's FFN input.
    if ffn_input is not None:
        u = ffn_input(rec)
    dense = [[_ffn(u[i], wts["w1"][e], wts["w2"][e], prm["gelu"]) for e in range(E)] for i in range(T)]
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
    ys = []
    copy = prm.get("token_reuse_policy", "current") == "copy" and not refresh
    for i in range(T):
        y = [0.0] * D
        for p in range(k):
            h = ch[i][slot[i][p]]
            for d in range(D):
                y[d] += w_cur[i][p] * h[d]
        if sh is not None:
            for d in range(D):
                y[d] += sh[i][d]
        if copy and not any(rec[i]):
            # Sec. 4.1 "reuse cached states": the token's last MoE output.
            y = list(state["cache_y"][i])
        ys.append(y)
        base = u[i] if resid is None else resid[i]
        g = [1.0] * D if gate is None else gate[i]
        out.append([base[d] + g[d] * y[d] for d in range(D)])
    cn = [[math.sqrt(sum(v * v for v in ch[i][q])) for q in range(k)] for i in range(T)]
    new = dict(cache_e=ce, cache_w=cw, cache_norm=cn, cache_h=ch, shared_h=sh, C=C, cache_y=ys)
    dec = dict(e=e_cur, w=w_cur, recompute=rec, slot=slot, tau=tau)
    return out, new, dec


def empty_state(T, D, E, k, n_shared):
    return dict(cache_e=[[-1] * k for _ in range(T)], cache_w=[[0.0] * k for _ in range(T)],
                cache_norm=[[0.0] * k for _ in range(T)],
                cache_h=[[[0.0] * D for _ in range(k)] for _ in range(T)],
                shared_h=[[0.0] * D for _ in range(T)] if n_shared else None,
                C=[[0.0] * T for _ in range(E)], cache_y=[[0.0] * D for _ in range(T)])


# ---------------------------------------------------------------------------
# AdaLN DiT-MoE block (Sec. 3 residual form, Sec. 4.1 cache)
# ---------------------------------------------------------------------------

def _silu(z: float) -> float:
    return z / (1.0 + math.exp(-z))


def _layer_norm_mod(v, shift, scale, eps):
    D = len(v)
    mean = sum(v) / D
    var = sum((a - mean) ** 2 for a in v) / D
    r = 1.0 / math.sqrt(var + eps)
    return [(v[d] - mean) * r * (1.0 + scale[d]) + shift[d] for d in range(D)]


def _attention_row(hq, keys_h, wts, H):
    """Attention output of one token over the rows keys_h of its sample."""
    D = len(hq)
    dh = D // H
    wq, bq = wts["w_qkv"], wts.get("b_qkv")

    def proj(row, r0):
        return [sum(float(wq[r0 + j][d]) * row[d] for d in range(D)) + (float(bq[r0 + j]) if bq is not None else 0.0)
                for j in range(D)]

    q = proj(hq, 0)
    ks = [proj(r, D) for r in keys_h]
    vs = [proj(r, 2 * D) for r in keys_h]
    A = [0.0] * D
    for hd in range(H):
        lo = hd * dh
        sc = [sum(q[lo + j] * kr[lo + j] for j in range(dh)) / math.sqrt(dh) for kr in ks]
        m = max(sc)
        ex = [math.exp(v - m) for v in sc]
        tot = sum(ex)
        for n, vr in enumerate(vs):
            for j in range(dh):
                A[lo + j] += ex[n] / tot * vr[lo + j]
    wo, bo = wts["w_o"], wts.get("b_o")
    return [sum(float(wo[j][d]) * A[d] for d in range(D)) + (float(bo[j]) if bo is not None else 0.0)
            for j in range(D)]


def adaln_block_step(state: dict, x, cond, wts: dict, prm: dict, refresh: bool):
    """One AdaLN block step; state adds attn_a [T][D].  prm adds n_heads,
    seq_len, attn_policy ("sync" / "stale" / "full") and ln_eps.  Returns
    (out, new_state, decisions) with decisions adding u, m and attn_rows."""
    T, D = len(x), len(x[0])
    S = prm["seq_len"] or T
    eps = prm["ln_eps"]
    x = [[float(v) for v in row] for row in x]
    # Six modulation vectors per sample from SiLU(c).
    mods = []
    for b in range(len(cond)):
        sc = [_silu(float(v)) for v in cond[b]]
        row = [sum(float(wts["w_ada"][j][d]) * sc[d] for d in range(D))
               + (float(wts["b_ada"][j]) if wts.get("b_ada") is not None else 0.0) for j in range(6 * D)]
        mods.append([row[f * D:(f + 1) * D] for f in range(6)])
    md = [mods[i // S] for i in range(T)]
    h = [_layer_norm_mod(x[i], md[i][0], md[i][1], eps) for i in range(T)]

    def attn(i):
        b = i // S
        return _attention_row(h[i], h[b * S:(b + 1) * S], wts, prm["n_heads"])

    full = refresh or prm["attn_policy"] == "full"
    a = [attn(i) for i in range(T)] if full else [list(r) for r in state["attn_a"]]
    u = [[x[i][d] + md[i][2][d] * a[i][d] for d in range(D)] for i in range(T)]
    m = [_layer_norm_mod(u[i], md[i][3], md[i][4], eps) for i in range(T)]
    route_in = [list(r) for r in m]
    rows = list(range(T)) if full else []

    def ffn_input(rec):
        if full or prm["attn_policy"] != "sync":
            return m
        for i in range(T):
            if any(rec[i]):
                rows.append(i)
                a[i] = attn(i)
                u[i] = [x[i][d] + md[i][2][d] * a[i][d] for d in range(D)]
                m[i] = _layer_norm_mod(u[i], md[i][3], md[i][4], eps)
        return m

    out, new, dec = layer_step(state, route_in, wts, prm, refresh, ffn_input=ffn_input, resid=u,
                               gate=[md[i][5] for i in range(T)])
    new["attn_a"] = a
    dec.update(u=u, m=m, attn_rows=rows)
    return out, new, dec
