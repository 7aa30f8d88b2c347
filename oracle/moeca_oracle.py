"""MoECa oracle: a plain, slow CPU statement of the branch-cached MoE layer.

TEST INFRASTRUCTURE.  Only the tests, the package smoke check and the CPU
baseline leg of the benchmark may import this module.  It shares no code with
the CUDA path.

Arithmetic is float64 (numpy).  Where floating point decides an integer -- the
top-k expert choice and the recompute/reuse decision -- the decision is taken
on values rounded to float32, the precision the GPU decides in; the other
quantities stay float64.  Matrix products use numpy's matmul as a library step.

Each function names the passage of the paper it follows:
  Eq. 5 / Eq. 6   routed (and shared) MoE-FFN output, residual form
  Eq. 7           routing set B_i^t and branch cache C_i^{t0}
  Sec. 4.1        full-computation vs cache steps, synchronized update rule
  Eq. 8           branch-level combine with current gate weights
  Sec. 4.2, Eq. 9 branch matching, score s = w + l1*Delta + l2*o, s > tau
  Eq. 10          EMA spatial activation statistic C_{e,i}
  Eq. 11          spatial response entropy H_e and its normalisation
  Eq. 12          expert-aware threshold tau_e = tau0 (1 + alpha (2 Hbar_e - 1))
  Sec. 4.1        attention output a_i cached with the branches; a token's
                  attention is recomputed on the step its recompute set is
                  non-empty (synchronized MoE / attention update)
  Table 4         "without sync. update": attention reused on every cache step
  Sec. 3, Eq. 2   DiT block: attention then MLP (MoE) sub-layer, each in the
                  residual form x + AdaLN o f(x)
  Sec. 3, Eq. 1   reverse transition of the sampler

Readings where the paper is silent (each is a switch in ``Params``):
  * gate weights: softmax over all E experts, top-k, then renormalised over
    the k picks (``renorm_topk``);
  * top-k order p: descending logit, ties to the lower expert id;
  * ||h|| in o is the L2 norm over D of the unweighted cached branch output,
    the sum runs over the token's k cached routed slots, o = 0 if it is 0;
  * Hbar_e = H_e / ln T over all T token rows ("log_t"); an expert with an
    all-zero statistic, or T = 1, gets Hbar = 0.5; "minmax" rescales
    H across the layer's experts instead;
  * C starts at 0 and is updated on every step, refresh steps included;
  * an unmatched branch takes a cache slot whose expert is no longer routed,
    in ascending p -> ascending q order; on a full-computation step slot = p;
  * a reused slot keeps its cached weight w^{t0} ("keep") or takes w^t
    ("overwrite");
  * shared experts are recomputed on full-computation steps and for tokens
    with a non-empty recompute set ("sync"), or always ("always");
  * Eq. 8 forms every token's output from its branches with the current
    gate weights w^t ("current"); Sec. 4.1's other wording, that a token
    with an empty recompute set reuses its cached state, is the "copy"
    reading: such a token takes its last computed MoE output y^{t0}
    unchanged (``token_reuse_policy``);
  * GELU is the tanh form ("tanh") or the erf form ("erf"); experts have no bias.
  * a DiT block (n_heads > 0) is x -> u = x + Attn(x) -> u + MoE(u), without
    normalisation or modulation; attention is multi-head self-attention over
    the seq_len consecutive token rows of each sample, with all of the
    sample's keys and values taken from the current block input;
  * on a cache step the recompute decision comes before the attention
    update, so the router sees u' = x + a^{t0} (cached attention output);
    a token with a non-empty recompute set then recomputes its attention,
    and its recomputed branches and its residual use u = x + a^t; a token
    without one keeps u' (``attn_policy`` "sync"); "stale" reuses a^{t0} on
    every cache step (Table 4's ablation); "full" recomputes attention for
    every token on every step and routes on the fresh input;
  * ``act_store`` "bf16" rounds the block's stored activations (a, u) to
    bfloat16, the storage type of the bf16 kernels, so that decisions taken
    on u' use the same input on both sides; "f64" keeps them exact.
  * an AdaLN block (``adaln``; Sec. 3 names AdaLN, the form is DiT's): per
    sample, SiLU(c) W_ada^T + b_ada gives shift, scale and gate for each
    sub-layer; a sub-layer reads LN(v) (1 + scale) + shift (LN over D, no
    affine, eps 1e-6) and is added as v + gate f; the caches hold ungated
    outputs and each step applies its own modulation; under the sync rule
    the router sees m' = modulate(LN(x + gate_a a^{t0})).
  * sampler (Eq. 1): linear betas 1e-4 .. 0.02 over 1000 training steps, a
    run of n steps visits n evenly spaced training steps (rounded half up),
    variance beta_t, no noise on the last step.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

_TINY = 1e-30


@dataclass
class Params:
    """Hyper-parameters of MoECa (Eq. 9, Eq. 10, Eq. 12, Sec. 5.1) and readings."""

    top_k: int
    lambda1: float = 1.0
    lambda2: float = 0.5
    tau0: float = 0.8
    alpha: float = 0.6
    beta: float = 0.65
    refresh_period: int = 0
    renorm_topk: bool = True
    entropy_norm: str = "log_t"        # or "minmax"
    shared_policy: str = "sync"        # or "always"
    reused_meta_policy: str = "keep"   # or "overwrite"
    gelu: str = "tanh"                 # or "erf"
    score_terms: int = 7               # Eq. 9 terms kept: 1 = w, 2 = lambda1 Delta, 4 = lambda2 o (Table 5)
    granularity: str = "branch"        # or "token": a token's k branches share one decision
    n_heads: int = 0                   # > 0: each layer is a DiT block with an attention sub-layer
    seq_len: int = 0                   # token rows per sample (attention scope); 0: all T rows
    attn_policy: str = "sync"          # or "stale" (Table 4 ablation) or "full"
    act_store: str = "f64"             # or "bf16": storage rounding of the block's a and u
    adaln: bool = False                # DiT block with AdaLN modulation of both sub-layers (Sec. 3)
    ln_eps: float = 1e-6               # layer-normalisation epsilon of the AdaLN block
    token_reuse_policy: str = "current"  # or "copy": R_i empty => y_i = y_i^{t0} (Sec. 4.1)


# ---------------------------------------------------------------------------
# Expert FFN (Eq. 5 / Eq. 6)
# ---------------------------------------------------------------------------

def gelu(z: np.ndarray, form: str = "tanh") -> np.ndarray:
    """GELU; the tanh form is the DiT convention, the erf form is exact GELU."""
    z = np.asarray(z, dtype=np.float64)
    if form == "tanh":
        return 0.5 * z * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (z + 0.044715 * z ** 3)))
    if form == "erf":
        from scipy.special import erf
        return 0.5 * z * (1.0 + erf(z / math.sqrt(2.0)))
    raise ValueError(form)


def expert_ffn(u_rows: np.ndarray, w1: np.ndarray, w2: np.ndarray, form: str) -> np.ndarray:
    """FFN_e(u) = W2_e GELU(W1_e u) for each row of ``u_rows``.

    w1 is [F, D] and w2 is [D, F] (rows are output features).
    """
    u = np.asarray(u_rows, dtype=np.float64)
    hmid = gelu(u @ np.asarray(w1, np.float64).T, form)
    return hmid @ np.asarray(w2, np.float64).T


# ---------------------------------------------------------------------------
# Attention path of a DiT block (Sec. 4.1)
# ---------------------------------------------------------------------------

def round_bf16(a) -> np.ndarray:
    """Nearest bfloat16 value of each element (ties to even), as float64.

    bfloat16 keeps the top 16 bits of a float32: the value is rounded to
    float32 first (exact for a sum of two bfloat16 values), then its low
    16 bits are rounded away.  Infinities and NaNs pass through.
    """
    f = np.ascontiguousarray(np.asarray(a, np.float64).astype(np.float32))
    bits = f.view(np.uint32).astype(np.uint64)
    keep = (bits >> 16) & 1
    r = ((bits + 0x7FFF + keep) & 0xFFFF0000).astype(np.uint32)
    out = r.view(np.float32).astype(np.float64)
    special = ~np.isfinite(f)
    out[special] = f[special]
    return out


def attention(x, w_qkv, b_qkv, w_o, b_o, n_heads: int, seq_len: int, rows=None) -> np.ndarray:
    """Multi-head self-attention output a_i of a DiT block (the a_i of Sec. 4.1).

    x is [T, D]; token rows come in samples of ``seq_len`` consecutive rows
    (0: one sample of T rows) and attend to every row of their own sample.
    w_qkv is [3D, D]: rows [0, D) give queries, [D, 2D) keys, [2D, 3D)
    values, head h owning rows [h dh, (h + 1) dh) of each (dh = D / n_heads);
    b_qkv [3D] and b_o [D] may be None.  Per head,
        A_h = softmax(Q_h K_h^T / sqrt(dh)) V_h   (softmax over the keys),
    the heads are concatenated and a = A w_o^T + b_o.  Returns a for the
    token rows ``rows`` (ascending ids; None: all), [len(rows), D].
    """
    x = np.asarray(x, np.float64)
    T, D = x.shape
    H = int(n_heads)
    dh = D // H
    S = int(seq_len) or T
    qkv = x @ np.asarray(w_qkv, np.float64).T
    if b_qkv is not None:
        qkv = qkv + np.asarray(b_qkv, np.float64)[None, :]
    q, k, v = qkv[:, :D], qkv[:, D:2 * D], qkv[:, 2 * D:]
    rows = np.arange(T) if rows is None else np.asarray(rows, np.int64)
    A = np.zeros((len(rows), D))
    for b in range(T // S):
        mine = np.nonzero(rows // S == b)[0]
        if len(mine) == 0:
            continue
        qi = rows[mine]
        keys = slice(b * S, (b + 1) * S)
        for h in range(H):
            hs = slice(h * dh, (h + 1) * dh)
            s = q[qi, hs] @ k[keys, hs].T / math.sqrt(dh)          # [n, S]
            p = np.exp(s - s.max(axis=1, keepdims=True))
            p /= p.sum(axis=1, keepdims=True)
            A[mine, hs] = p @ v[keys, hs]
    a = A @ np.asarray(w_o, np.float64).T
    if b_o is not None:
        a = a + np.asarray(b_o, np.float64)[None, :]
    return a


# ---------------------------------------------------------------------------
# Routing (Eq. 7)
# ---------------------------------------------------------------------------

def router_logits(u: np.ndarray, w_gate: np.ndarray, b_gate=None) -> np.ndarray:
    """Gate logits u W_g^T (+ b), float64, [T, E]."""
    z = np.asarray(u, np.float64) @ np.asarray(w_gate, np.float64).T
    if b_gate is not None:
        z = z + np.asarray(b_gate, np.float64)[None, :]
    return z


def route(u, w_gate, b_gate, k: int, renorm: bool):
    """Top-k routing set B_i^t = {(e_p, w_p)}, p = 1..k (Eq. 7).

    Returns (e [T,k] int32, w [T,k] float64, near [T] float64, cond [T]) where
    ``near`` is the smallest gap between adjacent ranks 1..k+1 of the float32
    logits relative to ``cond``, the token's largest sum_d |u_d W_ed| (+|b_e|):
    the magnitude a float32 dot product accumulates, which sets its rounding.
    """
    z = router_logits(u, w_gate, b_gate)
    cond = np.abs(np.asarray(u, np.float64)) @ np.abs(np.asarray(w_gate, np.float64)).T
    if b_gate is not None:
        cond = cond + np.abs(np.asarray(b_gate, np.float64))[None, :]
    cond = np.maximum(cond.max(axis=1), _TINY)
    T, E = z.shape
    if not (1 <= k <= E):
        raise ValueError("top_k must be in [1, E]")
    z32 = z.astype(np.float32)
    # Descending float32 logit; the stable sort keeps ties in ascending expert id.
    order = np.argsort(-z32, axis=1, kind="stable")
    e_sel = order[:, :k].astype(np.int32)
    zmax = z.max(axis=1, keepdims=True)
    p_all = np.exp(z - zmax)
    p_all /= p_all.sum(axis=1, keepdims=True)
    w = np.take_along_axis(p_all, e_sel.astype(np.int64), axis=1)
    if renorm:
        w = w / w.sum(axis=1, keepdims=True)
    ranks = min(k + 1, E)
    zs = np.take_along_axis(z32.astype(np.float64), order[:, :ranks], axis=1)
    if ranks > 1:
        near = (zs[:, :-1] - zs[:, 1:]).min(axis=1) / cond
    else:
        near = np.full(T, np.inf)
    return e_sel, w, near, cond


# ---------------------------------------------------------------------------
# Expert-aware adaptive threshold (Eq. 10 - Eq. 12)
# ---------------------------------------------------------------------------

def ema_update(C: np.ndarray, e_sel: np.ndarray, beta: float) -> np.ndarray:
    """C_{e,i} <- beta C_{e,i} + (1 - beta) 1[e in B_i]   (Eq. 10).  C is [E, T]."""
    E, T = C.shape
    ind = np.zeros((E, T), dtype=np.float64)
    for i in range(T):
        for e in e_sel[i]:
            ind[int(e), i] = 1.0
    return beta * np.asarray(C, np.float64) + (1.0 - beta) * ind


def spatial_entropy(C: np.ndarray) -> np.ndarray:
    """H_e = -sum_i P_e(i) log P_e(i), P_e(i) = C_{e,i} / sum_j C_{e,j}  (Eq. 11).

    Terms with P = 0 contribute 0.  Experts with an all-zero row get NaN.
    """
    C = np.asarray(C, np.float64)
    E, T = C.shape
    H = np.full(E, np.nan)
    for e in range(E):
        S = C[e].sum()
        if S <= 0.0:
            continue
        P = C[e] / S
        nz = P > 0.0
        H[e] = -np.sum(P[nz] * np.log(P[nz]))
    return H


def normalized_entropy(C: np.ndarray, mode: str = "log_t") -> np.ndarray:
    """Hbar_e in [0, 1] (Eq. 11 normalisation); see the module readings."""
    E, T = C.shape
    H = spatial_entropy(C)
    live = ~np.isnan(H)
    Hbar = np.full(E, 0.5)
    if mode == "log_t":
        if T > 1:
            Hbar[live] = np.clip(H[live] / math.log(T), 0.0, 1.0)
    elif mode == "minmax":
        if live.any():
            lo, hi = H[live].min(), H[live].max()
            if hi > lo:
                Hbar[live] = (H[live] - lo) / (hi - lo)
    else:
        raise ValueError(mode)
    return Hbar


def expert_threshold(Hbar: np.ndarray, tau0: float, alpha: float) -> np.ndarray:
    """tau_e = tau0 (1 + alpha (2 Hbar_e - 1))   (Eq. 12)."""
    return tau0 * (1.0 + alpha * (2.0 * np.asarray(Hbar, np.float64) - 1.0))


# ---------------------------------------------------------------------------
# Branch matching, scoring and the recompute set (Sec. 4.2, Eq. 9)
# ---------------------------------------------------------------------------

def historical_contribution(cache_norm: np.ndarray) -> np.ndarray:
    """o_{i,q} = ||h_{i,q}|| / sum_j ||h_{i,j}||  (Eq. 9); 0 where the sum is 0."""
    n = np.asarray(cache_norm, np.float64)
    s = n.sum(axis=1, keepdims=True)
    return np.where(s > 0.0, n / np.where(s > 0.0, s, 1.0), 0.0)


def select_branches(e_cur, w_cur, cache_e, cache_w, cache_norm, tau, lambda1, lambda2,
                    refresh: bool, score_terms: int = 7, granularity: str = "branch"):
    """Partition B_i^t into the recompute set R_i^t and the reuse set.

    Eq. 9 scores a matched branch with s = w + lambda1 Delta + lambda2 o;
    `score_terms` keeps a subset of the three terms (the signal ablation of
    Table 5: bit 1 = w, 2 = lambda1 Delta, 4 = lambda2 o).  With granularity
    "token", a token's k branches share one decision, as in token-level
    caching (Sec. 3): all of them are recomputed when the branch rule would
    recompute any of them, else all are reused.

    Returns a dict of [T, k] arrays:
      recompute (bool), slot (int32: cache slot that holds branch p after the
      step), matched (bool), score (float64, NaN if unmatched) and margin
      (|s - tau| / |tau|, inf where no threshold decides; in token mode the
      smallest margin of the token, which decides all its branches).
    """
    e_cur = np.asarray(e_cur)
    T, k = e_cur.shape
    recompute = np.ones((T, k), dtype=bool)
    slot = np.tile(np.arange(k, dtype=np.int32), (T, 1))
    matched = np.zeros((T, k), dtype=bool)
    score = np.full((T, k), np.nan)
    margin = np.full((T, k), np.inf)
    if refresh:
        return dict(recompute=recompute, slot=slot, matched=matched, score=score, margin=margin)
    o = historical_contribution(cache_norm)
    tau = np.asarray(tau, np.float64)
    for i in range(T):
        q_of = [-1] * k
        for p in range(k):
            e = int(e_cur[i, p])
            hits = [q for q in range(k) if int(cache_e[i, q]) == e]
            if not hits:
                continue          # unmatched: no cached state for this expert
            q = hits[0]
            q_of[p] = q
            matched[i, p] = True
            w = float(w_cur[i, p])
            delta = abs(w - float(cache_w[i, q]))
            s = ((w if score_terms & 1 else 0.0)
                 + (lambda1 * delta if score_terms & 2 else 0.0)
                 + (lambda2 * float(o[i, q]) if score_terms & 4 else 0.0))
            score[i, p] = s
            t = float(tau[e])
            recompute[i, p] = bool(np.float32(s) > np.float32(t))
            if math.isfinite(t):
                margin[i, p] = abs(s - t) / max(abs(t), _TINY)
        if granularity == "token":
            if recompute[i].any():
                recompute[i, :] = True
            margin[i, :] = margin[i].min()
        # Matched branches keep their slot; unmatched ones take the freed slots.
        free = [q for q in range(k) if q not in q_of]
        unmatched = [p for p in range(k) if q_of[p] < 0]
        for p in range(k):
            if q_of[p] >= 0:
                slot[i, p] = q_of[p]
        for p, q in zip(unmatched, free):
            slot[i, p] = q
    return dict(recompute=recompute, slot=slot, matched=matched, score=score, margin=margin)


# ---------------------------------------------------------------------------
# Layer state and one step of a layer
# ---------------------------------------------------------------------------

@dataclass
class LayerState:
    """Per-layer cache (Eq. 7) and EMA statistic (Eq. 10) for T token rows."""

    cache_e: np.ndarray        # [T, k] int32   e_{i,q}^{t0}
    cache_w: np.ndarray        # [T, k] float64 w_{i,q}^{t0}
    cache_norm: np.ndarray     # [T, k] float64 ||h_{i,q}^{t0}||
    cache_h: np.ndarray        # [T, k, D] float64 h_{i,q}^{t0}
    shared_h: np.ndarray | None  # [T, D] float64, shared-expert output
    C: np.ndarray              # [E, T] float64 C_{e,i}
    valid: bool = False
    attn_a: np.ndarray | None = None  # [T, D] float64 a_i^{t0} of a DiT block (Sec. 4.1)
    cache_y: np.ndarray | None = None  # [T, D] float64 y_i^{t0}, the token's last MoE output (ungated)

    @staticmethod
    def empty(T: int, D: int, E: int, k: int, n_shared: int, attention: bool = False) -> "LayerState":
        return LayerState(
            cache_e=np.full((T, k), -1, np.int32), cache_w=np.zeros((T, k)),
            cache_norm=np.zeros((T, k)), cache_h=np.zeros((T, k, D)),
            shared_h=np.zeros((T, D)) if n_shared else None, C=np.zeros((E, T)), valid=False,
            attn_a=np.zeros((T, D)) if attention else None, cache_y=np.zeros((T, D)))

    def copy(self) -> "LayerState":
        return LayerState(self.cache_e.copy(), self.cache_w.copy(), self.cache_norm.copy(),
                          self.cache_h.copy(), None if self.shared_h is None else self.shared_h.copy(),
                          self.C.copy(), self.valid, None if self.attn_a is None else self.attn_a.copy(),
                          None if self.cache_y is None else self.cache_y.copy())


def recompute_and_combine(state: LayerState, u: np.ndarray, e_cur, w_cur, rec, slot, weights: dict,
                          prm: Params, refresh: bool, resid=None, gate=None):
    """Apply a recompute decision and form the layer output (Sec. 4.1, Eq. 5-8).

    Recomputes FFN_e(u_i) for the branches in R (rows of one expert together),
    stores them in their cache slots with (e^t, w^t), recomputes shared experts
    under the synchronized rule, combines every branch p from slot(p) with the
    current weight w^t (Eq. 8), adds the residual and refreshes the cached
    norms.  Returns (out [T, D], new state, token_any [T]).

    ``resid`` and ``gate`` ([T, D], or None) give the AdaLN block's output
    resid + gate * y (Sec. 3 residual form) instead of u + y.

    Under ``token_reuse_policy`` "copy", a token with an empty recompute set
    on a cache step takes y_i = y_i^{t0}, its MoE output of the last step it
    computed one (Sec. 4.1, "reuse cached states"), in place of Eq. 8 with
    the current weights.  The new state keeps every token's y (ungated).
    """
    u = np.asarray(u, np.float64)
    T, D = u.shape
    k = prm.top_k
    new = state.copy()
    e_cur = np.asarray(e_cur)
    rec = np.asarray(rec, bool)
    slot = np.asarray(slot)
    for e in np.unique(e_cur[rec]):
        rows = np.argwhere(rec & (e_cur == e))
        h = expert_ffn(u[rows[:, 0]], weights["w1"][e], weights["w2"][e], prm.gelu)
        for (i, p), hv in zip(rows, h):
            q = slot[i, p]
            new.cache_h[i, q] = hv
            new.cache_e[i, q] = e
            new.cache_w[i, q] = w_cur[i, p]
    if prm.reused_meta_policy == "overwrite":
        for i, p in np.argwhere(~rec):
            new.cache_w[i, slot[i, p]] = w_cur[i, p]
    token_any = rec.any(axis=1)
    ws1 = weights.get("ws1")
    if ws1 is not None and len(ws1):
        if refresh or prm.shared_policy == "always":
            rows = np.arange(T)
        else:
            rows = np.nonzero(token_any)[0]
        if len(rows):
            acc = np.zeros((len(rows), D))
            for s in range(len(ws1)):
                acc += expert_ffn(u[rows], ws1[s], weights["ws2"][s], prm.gelu)
            new.shared_h[rows] = acc
    # Eq. 8: every current branch p reads slot(p), fresh or cached, with w^t.
    y = np.zeros((T, D))
    for p in range(k):
        y += np.asarray(w_cur, np.float64)[:, p:p + 1] * new.cache_h[np.arange(T), slot[:, p]]
    if new.shared_h is not None:
        y += new.shared_h
    if prm.token_reuse_policy == "copy" and not refresh:
        if state.cache_y is None:
            raise ValueError("the copy reading needs the cached outputs y^{t0}")
        keep = ~token_any
        y[keep] = state.cache_y[keep]
    elif prm.token_reuse_policy not in ("current", "copy"):
        raise ValueError(prm.token_reuse_policy)
    new.cache_y = y.copy()
    if gate is not None:
        y = np.asarray(gate, np.float64) * y
    out = (u if resid is None else np.asarray(resid, np.float64)) + y
    new.cache_norm = np.sqrt(np.sum(new.cache_h ** 2, axis=2))
    new.valid = True
    return out, new, token_any


def layer_step(state: LayerState, u: np.ndarray, weights: dict, prm: Params, refresh: bool):
    """One MoE layer at one denoising step; returns (out [T, D], new state, info).

    Order of work: route (Eq. 7) -> EMA (Eq. 10) -> entropy and tau (Eq. 11-12)
    -> match, score, decide (Eq. 9) -> recompute R (Eq. 5) -> shared experts
    under the synchronized rule (Sec. 4.1) -> combine with current gate weights
    (Eq. 8) plus the residual (Eq. 5 / 6) -> refresh the cached norms.
    """
    info = decide(state, u, weights, prm, refresh)
    out, new, token_any = recompute_and_combine(state, u, info["e"], info["w"], info["recompute"],
                                                info["slot"], weights, prm, refresh)
    new.C = info["C"]
    info["token_any"] = token_any
    return out, new, info


def decide(state: LayerState, u: np.ndarray, weights: dict, prm: Params, refresh: bool) -> dict:
    """The decision half of a layer step, taken on the router input u:
    route (Eq. 7) -> EMA (Eq. 10) -> entropy and tau (Eq. 11-12) -> match,
    score, decide and assign slots (Sec. 4.2, Eq. 9).  Returns the routing,
    the new statistic C, tau and the select_branches fields."""
    u = np.asarray(u, np.float64)
    k = prm.top_k
    e_cur, w_cur, near, _ = route(u, weights["w_gate"], weights.get("b_gate"), k, prm.renorm_topk)
    C = ema_update(state.C, e_cur, prm.beta)
    Hbar = normalized_entropy(C, prm.entropy_norm)
    tau = expert_threshold(Hbar, prm.tau0, prm.alpha)
    sel = select_branches(e_cur, w_cur, state.cache_e, state.cache_w, state.cache_norm, tau,
                          prm.lambda1, prm.lambda2, refresh, prm.score_terms, prm.granularity)
    return dict(e=e_cur, w=w_cur, near_route=near, C=C, Hbar=Hbar, tau=tau,
                token_any=sel["recompute"].any(axis=1), refresh=refresh, **sel)


def block_step(state: LayerState, x: np.ndarray, weights: dict, prm: Params, refresh: bool):
    """One DiT-MoE block at one denoising step: the attention sub-layer, then
    the MoE sub-layer, with the attention output a_i cached beside the
    branches (Sec. 4.1).  Returns (out [T, D], new state, info).

    Full-computation step, or attn_policy "full": a = Attn(x) for every
    token, u = x + a, and the MoE layer step runs on u.
    Cache step, "sync" (Sec. 4.1): the decision is taken on u' = x + a^{t0};
    tokens with a non-empty recompute set recompute a_i from the current x
    (all keys of their sample), store it, and take u_i = x_i + a_i; the
    others keep u'_i.  The recomputed branches take u as their input, Eq. 8
    combines with the gate weights routed on u', and the residual adds u.
    Cache step, "stale" (Table 4, without sync update): u = x + a^{t0} for
    every token and a is left as it is.
    ``info`` adds u (MoE input), route_in (router input) and attn_rows.
    """
    x = np.asarray(x, np.float64)
    T, D = x.shape
    store = round_bf16 if prm.act_store == "bf16" else (lambda v: np.asarray(v, np.float64))

    def attn(rows=None):
        return attention(x, weights["w_qkv"], weights.get("b_qkv"), weights["w_o"], weights.get("b_o"),
                         prm.n_heads, prm.seq_len, rows)

    if refresh or prm.attn_policy == "full":
        a = store(attn())
        u = store(x + a)
        out, new, info = layer_step(state, u, weights, prm, refresh)
        new.attn_a = a
        info.update(u=u, route_in=u, attn_rows=np.arange(T))
        return out, new, info
    u_pre = store(x + state.attn_a)
    if prm.attn_policy == "stale":
        out, new, info = layer_step(state, u_pre, weights, prm, refresh)
        new.attn_a = state.attn_a.copy()
        info.update(u=u_pre, route_in=u_pre, attn_rows=np.zeros(0, np.int64))
        return out, new, info
    if prm.attn_policy != "sync":
        raise ValueError(prm.attn_policy)
    info = decide(state, u_pre, weights, prm, refresh)
    rows = np.nonzero(info["token_any"])[0]
    a = state.attn_a.copy()
    u = u_pre.copy()
    if len(rows):
        a[rows] = store(attn(rows))
        u[rows] = store(x[rows] + a[rows])
    out, new, token_any = recompute_and_combine(state, u, info["e"], info["w"], info["recompute"],
                                                info["slot"], weights, prm, refresh)
    new.C = info["C"]
    new.attn_a = a
    info.update(u=u, route_in=u_pre, attn_rows=rows)
    return out, new, info


# ---------------------------------------------------------------------------
# DiT-MoE block with AdaLN modulation (Sec. 3, Eq. 2) and the sampler (Eq. 1)
# ---------------------------------------------------------------------------

def silu(z: np.ndarray) -> np.ndarray:
    """SiLU(z) = z / (1 + exp(-z)), the activation before the AdaLN projection."""
    z = np.asarray(z, np.float64)
    return z / (1.0 + np.exp(-z))


def layer_norm(v: np.ndarray, eps: float) -> np.ndarray:
    """Normalisation of each row over its D features, without affine
    parameters: (v - mean) / sqrt(var + eps), var the biased row variance."""
    v = np.asarray(v, np.float64)
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).mean(axis=-1, keepdims=True)
    return (v - mu) / np.sqrt(var + eps)


def adaln_modulation(c: np.ndarray, w_ada: np.ndarray, b_ada=None) -> np.ndarray:
    """The six AdaLN vectors of one block for every sample (Sec. 3).

    c is [B, D], one conditioning vector per sample (timestep and class
    embedding); w_ada is [6D, D] and b_ada [6D] or None.  Returns
    mod [B, 6, D] = reshape(SiLU(c) w_ada^T + b_ada): along axis 1 the
    attention sub-layer's shift, scale and gate, then the MoE sub-layer's.
    """
    c = np.asarray(c, np.float64)
    B, D = c.shape
    mod = silu(c) @ np.asarray(w_ada, np.float64).T
    if b_ada is not None:
        mod = mod + np.asarray(b_ada, np.float64)[None, :]
    return mod.reshape(B, 6, D)


def modulate(v: np.ndarray, shift: np.ndarray, scale: np.ndarray) -> np.ndarray:
    """AdaLN's affine map of a normalised row: v (1 + scale) + shift."""
    return np.asarray(v, np.float64) * (1.0 + np.asarray(scale, np.float64)) + np.asarray(shift, np.float64)


def token_rows(vec: np.ndarray, T: int, seq_len: int) -> np.ndarray:
    """Expand per-sample rows [B, D] to token rows [T, D] (samples of seq_len rows)."""
    S = int(seq_len) or T
    vec = np.asarray(vec, np.float64)
    if vec.shape[0] * S != T:
        raise ValueError("n_tokens must be n_samples * seq_len")
    return np.repeat(vec, S, axis=0)


def adaln_block_step(state: LayerState, x: np.ndarray, mod: np.ndarray, weights: dict, prm: Params,
                     refresh: bool):
    """One DiT-MoE block with AdaLN modulation at one denoising step (Sec. 3
    residual form, cached under Sec. 4.1).  mod is the block's [B, 6, D]
    output of ``adaln_modulation``.  Returns (out [T, D], new state, info).

        h = modulate(LN(x), shift_a, scale_a)          attention input
        a = Attn(h)                                     (cached: a^{t0})
        u = x + gate_a a
        m = modulate(LN(u), shift_m, scale_m)          MoE input
        out = u + gate_m y,  y of Eq. 8 on m

    The caches hold the ungated a and branch outputs; every step applies
    its own modulation.  Full-computation step, or attn_policy "full": a
    for every token, routed on m.  Cache step, "sync": the decision is taken
    on m' = modulate(LN(u'), ...) with u' = x + gate_a a^{t0}; tokens with a
    non-empty recompute set recompute a_i (all keys of their sample, from
    the current h), u_i and m_i, and their branches read m_i; the others
    keep u'_i and m'_i.  "stale": u' and m' for every token, a kept.
    ``info`` adds h, u (residual), m (FFN input), route_in and attn_rows.
    """
    x = np.asarray(x, np.float64)
    T, D = x.shape
    S = prm.seq_len or T
    mod = np.asarray(mod, np.float64)
    sh_a, sc_a, g_a, sh_m, sc_m, g_m = (token_rows(mod[:, j], T, S) for j in range(6))
    store = round_bf16 if prm.act_store == "bf16" else (lambda v: np.asarray(v, np.float64))
    eps = prm.ln_eps
    h = store(modulate(layer_norm(x, eps), sh_a, sc_a))

    def attn(rows=None):
        return attention(h, weights["w_qkv"], weights.get("b_qkv"), weights["w_o"], weights.get("b_o"),
                         prm.n_heads, prm.seq_len, rows)

    def moe_input(u, rows):
        return store(modulate(layer_norm(u, eps), sh_m[rows], sc_m[rows]))

    every = np.arange(T)
    if refresh or prm.attn_policy == "full":
        a = store(attn())
        u = store(x + g_a * a)
        m = moe_input(u, every)
        route_in, rows = m, every
    else:
        u = store(x + g_a * state.attn_a)
        m = moe_input(u, every)
        route_in = m
        a = state.attn_a.copy()
        rows = np.zeros(0, np.int64)
    info = decide(state, route_in, weights, prm, refresh)
    if not (refresh or prm.attn_policy == "full"):
        if prm.attn_policy == "sync":
            rows = np.nonzero(info["token_any"])[0]
            if len(rows):
                m = m.copy()
                u = u.copy()
                a[rows] = store(attn(rows))
                u[rows] = store(x[rows] + g_a[rows] * a[rows])
                m[rows] = moe_input(u[rows], rows)
        elif prm.attn_policy != "stale":
            raise ValueError(prm.attn_policy)
    out, new, token_any = recompute_and_combine(state, m, info["e"], info["w"], info["recompute"],
                                                info["slot"], weights, prm, refresh, resid=u, gate=g_m)
    new.C = info["C"]
    new.attn_a = a
    info.update(h=h, u=u, m=m, route_in=route_in, attn_rows=rows, token_any=token_any)
    return out, new, info


def ddpm_schedule(n_steps: int, n_train: int = 1000, beta_start: float = 1e-4, beta_end: float = 0.02):
    """Per-step coefficients of Eq. 1 for a sampling run of ``n_steps`` steps.

    The training schedule is beta_s linear from beta_start to beta_end over
    n_train steps, abar_s = prod_{r <= s} (1 - beta_r).  A run of n steps
    visits the training steps t_j = floor(j (n_train - 1) / (n_steps - 1) + 1/2),
    j = 0 .. n - 1, and takes abar'_j = abar_{t_j},
    alpha'_j = abar'_j / abar'_{j-1} (abar'_{-1} = 1), beta'_j = 1 - alpha'_j.
    Returns (t, alpha, alpha_bar, beta), each [n_steps], in j order (a run
    goes from j = n - 1 down to 0).
    """
    if n_steps < 2 or n_steps > n_train:
        raise ValueError("2 <= n_steps <= n_train")
    betas = np.linspace(beta_start, beta_end, n_train, dtype=np.float64)
    abar = np.cumprod(1.0 - betas)
    t = np.floor(np.arange(n_steps) * (n_train - 1) / (n_steps - 1) + 0.5).astype(np.int64)
    ab = abar[t]
    prev = np.concatenate([[1.0], ab[:-1]])
    alpha = ab / prev
    return t, alpha, ab, 1.0 - alpha


def ddpm_step(x_t, eps, z, alpha_t: float, alpha_bar_t: float, sigma_t: float) -> np.ndarray:
    """One reverse transition of Eq. 1: the mean
    (x_t - (1 - alpha_t) / sqrt(1 - abar_t) eps) / sqrt(alpha_t), plus sigma_t z.
    Eq. 1's variance is beta_t I, so sigma_t = sqrt(beta_t); the last step
    of a run (j = 0) takes sigma = 0 and returns the mean.  z is the
    standard normal draw, an input."""
    x_t = np.asarray(x_t, np.float64)
    mean = (x_t - (1.0 - alpha_t) / math.sqrt(1.0 - alpha_bar_t) * np.asarray(eps, np.float64)) / math.sqrt(alpha_t)
    return mean + sigma_t * np.asarray(z, np.float64)


def stats_of(info: dict) -> dict:
    """Branch counts of one layer step (Fig. 8's reuse-over-match ratio inputs)."""
    rec, matched = info["recompute"], info["matched"]
    return dict(branches=int(rec.size), matched=int(matched.sum()),
                recomputed=int(rec.sum()), reused=int((~rec).sum()),
                tokens_fully_reused=int((~info["token_any"]).sum()))


class Stack:
    """A stack of L MoE layers (DiT-MoE blocks when n_heads > 0) run over
    denoising steps (Sec. 4.1 schedule).

    A step is a full-computation step when it is forced, when the caches are
    not valid or the token count changed, or when ``refresh_period`` N > 0
    divides the step index; otherwise it is a cache step.
    """

    def __init__(self, layers: list, prm: Params, hidden: int, n_experts: int, n_shared: int = 0):
        self.layers = layers
        self.prm = prm
        self.D, self.E, self.S = hidden, n_experts, n_shared
        self.states = None
        self.T = None

    def is_refresh(self, step_index: int, n_tokens: int, force: bool = False) -> bool:
        N = self.prm.refresh_period
        return bool(force or self.states is None or n_tokens != self.T
                    or not all(s.valid for s in self.states)
                    or (N > 0 and step_index % N == 0))

    def step(self, x: np.ndarray, step_index: int, force: bool = False, cond=None):
        """One denoising step of the stack; ``cond`` [B, D] is the per-sample
        conditioning of AdaLN blocks (``prm.adaln``)."""
        x = np.asarray(x, np.float64)
        T = x.shape[0]
        refresh = self.is_refresh(step_index, T, force)
        if self.states is None or T != self.T:
            self.states = [LayerState.empty(T, self.D, self.E, self.prm.top_k, self.S, self.prm.n_heads > 0)
                           for _ in self.layers]
            self.T = T
        infos = []
        step_fn = block_step if self.prm.n_heads > 0 else layer_step
        for l, w in enumerate(self.layers):
            if self.prm.adaln:
                mod = adaln_modulation(cond, w["w_ada"], w.get("b_ada"))
                x, self.states[l], info = adaln_block_step(self.states[l], x, mod, w, self.prm, refresh)
                info["mod"] = mod
            else:
                x, self.states[l], info = step_fn(self.states[l], x, w, self.prm, refresh)
            infos.append(info)
        return x, infos
