"""Helpers for the GPU parity tests: run the CUDA stack and check every layer of
every step against the oracle, stage by stage (teacher forcing).

For each layer the oracle gets what the GPU had at the start of that stage:
  router    the layer input            -> top-k ids (exact unless near a tie),
                                          weights, EMA statistic, tau_e
  select    the GPU routing, tau and     -> recompute mask (exact unless
            the pre-step cache              |s - tau| < 1e-5 |tau|), slots,
                                            matched flags (exact)
  compact   the GPU mask                  -> per-group row lists (exact)
  FFN and   the GPU decisions and the     -> layer output, fresh cache rows
  combine   pre-step cache                   (tolerance), kept rows (exact)
A DiT-MoE block (n_heads > 0) first checks its attention sub-layer:
  attention the GPU block input x         -> recomputed a rows (tolerance), kept
                                             a rows (exact), u = bf16(x + a) (exact)
and the router check then takes the input the rule routes on: u on full
steps (and under the "stale" and "full" policies), bf16(x + a^{t0}) on a
sync cache step.
An AdaLN block (adaln = 1) checks instead:
  modulation the step's conditioning     -> six vectors per sample (tolerance)
  attention  the GPU x and modulation    -> h = LN-modulate(x), recomputed a rows
                                            (tolerance), kept a rows (exact)
  residual   the GPU a                    -> u = bf16(x + g_a a) (within one bf16
                                            step on a few elements)
  MoE input  the GPU u                    -> m, and the router input m' (same bound)
and the MoE check then routes on the GPU's router input, recomputes on m and
forms u + g_m y.
"""
from __future__ import annotations

import math
import os
from dataclasses import dataclass, field

import numpy as np

from oracle import moeca_oracle as O

NEAR = 1e-5
REPORTS = []  # (test id, Report) of every checked trajectory, for the session summary


def np_of(t):
    import torch
    if t is None:
        return None
    if t.dtype == torch.bfloat16:
        t = t.float()
    return t.cpu().numpy()


def rel_l2(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-30))


@dataclass
class Report:
    steps: int = 0
    layers_checked: int = 0
    tokens_routed: int = 0      # token rows whose routing was checked
    gaps_routed: int = 0        # adjacent-rank logit gaps those tokens have (min(k, E - 1) each)
    near_route: int = 0         # excluded: top-(k+1) logit gap < 1e-5 cond
    near_route_logit: int = 0   # the same gap < 1e-5 max|logit| (the window the library counts)
    near_route_diff: int = 0    # excluded tokens whose top-k ids actually differ
    near_score: int = 0         # excluded: |s - tau| < 1e-5 |tau|
    near_score_diff: int = 0    # excluded branches whose decision actually differs
    lib_near_route: int = 0     # the library's own counters (moeca_stats)
    lib_near_score: int = 0
    max_out: float = 0.0        # largest |output| checked
    widened: int = 0            # output elements whose bound exceeds 5e-2 (see output_abs_bound)
    branches: int = 0
    recomputed: int = 0
    reused: int = 0
    unmatched: int = 0
    attn_rows: int = 0
    tokens_copied: int = 0
    max_attn_rel_l2: float = 0.0
    max_rel_l2: float = 0.0
    max_abs: float = 0.0
    notes: list = field(default_factory=list)

    def summary(self) -> str:
        return (f"{self.steps} steps, {self.layers_checked} layer steps, {self.tokens_routed} tokens routed, "
                f"{self.branches} branches: near ties {self.near_route} (|logit| window {self.near_route_logit}, "
                f"library {self.lib_near_route}, differing {self.near_route_diff}), near threshold "
                f"{self.near_score} (library {self.lib_near_score}, differing {self.near_score_diff}); "
                f"max rel L2 {self.max_rel_l2:.2e}, max abs {self.max_abs:.2e} at max |out| {self.max_out:.1f} "
                f"({self.widened} elements with a bound above 5e-2)")


def params_of(cfg) -> O.Params:
    return O.Params(
        top_k=cfg.top_k, lambda1=cfg.lambda1, lambda2=cfg.lambda2, tau0=cfg.tau0, alpha=cfg.alpha,
        beta=cfg.beta, refresh_period=cfg.refresh_period, renorm_topk=bool(cfg.renorm_topk),
        entropy_norm="log_t" if cfg.entropy_norm == 0 else "minmax",
        shared_policy="sync" if cfg.shared_policy == 0 else "always",
        reused_meta_policy="keep" if cfg.reused_meta_policy == 0 else "overwrite",
        gelu="tanh" if cfg.gelu_tanh else "erf", score_terms=cfg.score_terms,
        granularity="branch" if cfg.granularity == 0 else "token",
        n_heads=cfg.n_heads, seq_len=cfg.seq_len, attn_policy=("sync", "stale", "full")[cfg.attn_policy],
        act_store="bf16" if cfg.dtype == 1 else "f64", adaln=bool(cfg.adaln), ln_eps=cfg.ln_eps,
        token_reuse_policy="copy" if cfg.token_reuse_policy else "current")


def oracle_weights(w: dict) -> dict:
    return {k: (None if v is None else np.asarray(v, np.float64)) for k, v in w.items()}


def state_to_oracle(st: dict | None, T, D, E, k, S) -> O.LayerState:
    if st is None or st["n_tokens"] == 0:
        return O.LayerState.empty(T, D, E, k, S)
    return O.LayerState(
        cache_e=np_of(st["cache_e"]).astype(np.int32), cache_w=np_of(st["cache_w"]).astype(np.float64),
        cache_norm=np_of(st["cache_norm"]).astype(np.float64), cache_h=np_of(st["cache_h"]).astype(np.float64),
        shared_h=None if st["shared_h"] is None else np_of(st["shared_h"]).astype(np.float64),
        C=np_of(st["ema"]).astype(np.float64).T.copy(), valid=True,
        cache_y=None if st.get("cache_y") is None else np_of(st["cache_y"]).astype(np.float64))


def gate_weight_tol(w_o, cond):
    """Tolerance of float32 gate weights against the float64 oracle.

    A float32 dot product over D terms misses the exact logit by about
    2^-24 * sum_d |u_d W_ed| (= cond); a softmax weight moves by at most
    2 w (1 - w) times a logit error.  8x that, plus 2e-6 of float32 softmax.
    """
    return 2e-6 + 8 * 2.0 ** -24 * cond[:, None] * 2 * w_o * (1 - w_o)


def check_gate_weights(w_g, w_o, cond):
    tol = gate_weight_tol(w_o, cond)
    err = np.abs(w_g - w_o)
    assert (err <= tol).all(), f"gate weights: worst err {err.max():.3e}, tol there {tol.flat[err.argmax()]:.3e}"


def expected_lists(e, rec, slot, token_any, E, k, n_shared, refresh, shared_always):
    """Rows of every expert group in ascending token order (the compaction's contract)."""
    T = e.shape[0]
    groups = [[] for _ in range(E + n_shared)]
    for i in range(T):
        for p in range(k):
            if rec[i, p]:
                groups[int(e[i, p])].append(i * k + int(slot[i, p]))
        if n_shared and (refresh or shared_always or token_any[i]):
            groups[E].append(i)
    counts = np.array([len(g) for g in groups], np.int32)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.int32)
    flat = np.array([r for g in groups for r in g], np.int32)
    return counts, offsets, flat


def check_attention(rep: Report, cfg, w: dict, pre: dict | None, post: dict, tr: dict, refresh: bool,
                    tol: float = 1e-2) -> np.ndarray:
    """Teacher-forced check of a DiT-MoE block's attention sub-layer (Sec. 4.1).

    bf16 storage of q, k, v, the softmax weights in the p v product and the
    attention rows bounds the relative L2 error of a fresh a row near 2^-8;
    ``tol`` allows a few times that.  Returns the router input the oracle
    must use for this layer."""
    wo = oracle_weights(w)
    x = np_of(tr["block_in"]).astype(np.float64)
    u = np_of(tr["layer_in"]).astype(np.float64)
    a_post = np_of(post["attn_a"]).astype(np.float64)
    T = x.shape[0]
    full = refresh or cfg.attn_policy == 2
    has_pre = pre is not None and pre["n_tokens"]
    a_pre = np_of(pre["attn_a"]).astype(np.float64) if has_pre else None
    if full:
        rows = np.arange(T)
    elif cfg.attn_policy == 1:
        rows = np.zeros(0, np.int64)
    else:
        rows = np.nonzero(np_of(tr["token_any"]))[0]
    if len(rows):
        a_o = O.attention(x, wo["w_qkv"], wo.get("b_qkv"), wo["w_o"], wo.get("b_o"), cfg.n_heads, cfg.seq_len, rows)
        rl = rel_l2(a_post[rows], a_o)
        rep.max_attn_rel_l2 = max(rep.max_attn_rel_l2, rl)
        assert rl <= tol, f"attention rows rel L2 {rl:.3e}"
        per_row = np.linalg.norm(a_post[rows] - a_o, axis=1) / np.maximum(np.linalg.norm(a_o, axis=1), 1e-30)
        assert per_row.max() <= 4 * tol, f"worst attention row rel L2 {per_row.max():.3e}"
    kept = np.setdiff1d(np.arange(T), rows)
    if len(kept):
        assert a_pre is not None, "a cache step without a cached attention output"
        assert np.array_equal(a_post[kept], a_pre[kept]), "kept attention rows changed"
    assert np.array_equal(u, O.round_bf16(x + a_post)), "MoE input u differs from bf16(x + a)"
    rep.attn_rows += len(rows)
    if full or cfg.attn_policy == 1:
        return u
    return O.round_bf16(x + a_pre)


def close_in_bf16(got, want, what: str, max_frac: float = 2e-3, floor=0.0):
    """``got`` (bf16 values from the GPU) equals bf16(``want``) except on a
    few elements, and there by at most one bf16 step plus ``floor``: the GPU
    rounds a float32 result, the oracle a float64 one, so values within
    float32 error of a bf16 rounding boundary may land on either side.
    ``floor`` (per element) is the float32 error of the result's ingredients,
    which dominates where a sum of larger terms nearly cancels."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    exact = O.round_bf16(want)
    diff = got != exact
    bound = np.maximum(np.abs(exact), 1e-30) * 2.0 ** -7 + np.broadcast_to(floor, exact.shape)
    off = np.abs(got - exact)
    bad = diff & (off > bound + 1e-30)
    assert not bad.any(), (f"{what}: {int(bad.sum())} elements off by more than one bf16 step, worst "
                           f"{off[bad].max():.3e} at |value| {np.abs(exact[bad][off[bad].argmax()]):.3e}")
    assert diff.mean() <= max_frac, f"{what}: {int(diff.sum())} of {diff.size} elements differ"
    return int(diff.sum())


def bf16_step(v):
    """Spacing of bfloat16 values at |v| (8 significant bits): 2^(floor(log2 |v|) - 7)."""
    a = np.maximum(np.abs(np.asarray(v, np.float64)), 2.0 ** -126)
    return 2.0 ** (np.floor(np.log2(a)) - 7)


def output_abs_bound(want, bf16: bool, terms=None):
    """Per-element max-abs bound of a layer output.

    bf16: 5e-2 (the stated bound), except where the rounding of the value
    itself and the rounding inside its freshly computed terms already exceed
    it.  There the bound is 1.5 bf16 steps of the value (the GPU rounds a
    float32 result, the oracle does not round) plus ``terms``, the worst-case
    bf16 error of the fresh branch outputs (``fresh_terms``).  float32: none
    (relative bounds only)."""
    if not bf16:
        return None
    b = 1.5 * bf16_step(want)
    if terms is not None:
        b = b + np.asarray(terms, np.float64)
    return np.maximum(5e-2, b)


def fresh_terms(u, wo: dict, e_g, w_g, rec, slot, new_o, gelu: str, gate=None, shared_rows=None):
    """Worst-case bf16 error, per output element, of the branch outputs
    computed this step (and the recomputed shared-expert row).

    A fresh h = bf16(sum_f W2_df hmid_f) with hmid = bf16(GELU(W1 u)) is off by
    at most 2^-9 sum_f |W2_df| |hmid_f| (each hidden activation rounded, all
    errors aligned) plus 2^-9 |h_d| (its own rounding); y weights it by
    |w_p|, and an AdaLN block's output by |gate|."""
    u = np.asarray(u, np.float64)
    T, D = u.shape
    terms = np.zeros((T, D))
    ch = new_o.cache_h

    def branch_err(rows, w1, w2):
        hm = np.abs(O.gelu(u[rows] @ np.asarray(w1, np.float64).T, gelu))
        return 2.0 ** -9 * (hm @ np.abs(np.asarray(w2, np.float64)).T)

    for e in np.unique(e_g[rec]):
        idx = np.argwhere(rec & (e_g == e))
        rows, ps = idx[:, 0], idx[:, 1]
        err = branch_err(rows, wo["w1"][e], wo["w2"][e]) + 2.0 ** -9 * np.abs(ch[rows, slot[rows, ps]])
        np.add.at(terms, rows, np.abs(w_g[rows, ps])[:, None] * err)
    ws1 = wo.get("ws1")
    if ws1 is not None and shared_rows is not None and new_o.shared_h is not None:
        rows = np.nonzero(np.asarray(shared_rows, bool))[0]
        if len(rows):
            w1s = ws1 if np.ndim(ws1) == 2 else ws1[0]
            w2s = wo["ws2"] if np.ndim(wo["ws2"]) == 2 else wo["ws2"][0]
            terms[rows] += branch_err(rows, w1s, w2s) + 2.0 ** -9 * np.abs(new_o.shared_h[rows])
    if gate is not None:
        terms *= np.abs(np.asarray(gate, np.float64))
    return terms


def check_output(rep: Report, got, want, bf16: bool, rel: float, what: str = "layer output", terms=None):
    """Relative L2 (global, and per token row within 4x) and, for bf16, the
    per-element max-abs bound of ``output_abs_bound``."""
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    rl = rel_l2(got, want)
    err = np.abs(got - want)
    rep.max_rel_l2 = max(rep.max_rel_l2, rl)
    rep.max_abs = max(rep.max_abs, float(err.max()) if err.size else 0.0)
    rep.max_out = max(rep.max_out, float(np.abs(want).max()) if want.size else 0.0)
    assert rl <= rel, f"{what} rel L2 {rl:.3e}"
    row_err = np.linalg.norm(got - want, axis=-1) / np.maximum(np.linalg.norm(want, axis=-1), 1e-30)
    worst = int(np.argmax(row_err))
    assert row_err.flat[worst] <= 4 * rel, f"{what} row {worst} rel L2 {row_err.flat[worst]:.3e}"
    bound = output_abs_bound(want, bf16, terms)
    if bound is not None:
        rep.widened += int((bound > 5e-2).sum())
        bad = err > bound
        if bad.any():
            j = int(np.argmax(np.where(bad, err - bound, -np.inf)))
            raise AssertionError(f"{what} max abs: {int(bad.sum())} elements over the bound, worst "
                                 f"{err.flat[j]:.3e} at |value| {abs(want.flat[j]):.3e} (bound {bound.flat[j]:.3e})")


def count_route_margins(rep: Report, u_route, wo: dict, k: int, renorm: bool, e_g):
    """Route on the oracle, count the near-tie tokens under both windows,
    and the excluded tokens whose ids actually differ.  Returns
    (e_o, w_o, ok, cond)."""
    e_o, w_o, near, cond = O.route(u_route, wo["w_gate"], wo.get("b_gate"), k, renorm)
    ok = near >= NEAR
    z = O.router_logits(u_route, wo["w_gate"], wo.get("b_gate"))
    zmax = np.maximum(np.abs(z).max(axis=1), 1e-30)
    rep.tokens_routed += len(ok)
    rep.gaps_routed += len(ok) * min(k, wo["w_gate"].shape[0] - 1)
    rep.near_route += int((~ok).sum())
    rep.near_route_logit += int((near * cond < NEAR * zmax).sum())
    rep.near_route_diff += int((~ok & (e_o != e_g).any(axis=1)).sum())
    return e_o, w_o, ok, cond


def assert_margins(rep: Report, max_frac: float = 5e-3):
    """The excluded entries are reported and bounded: near-tie tokens are at
    most ``max_frac`` of the adjacent-rank gaps checked (a top-8 token has
    eight chances to tie), near-threshold branches at most ``max_frac`` of
    the branches (plus two each), and of the excluded entries at most a few
    actually disagree -- a disagreement needs a gap near the float32
    rounding of the dot product, about 1e-7 of cond, a hundredth of the
    window."""
    assert rep.near_route <= max_frac * rep.gaps_routed + 2, f"near-tie tokens: {rep.summary()}"
    assert rep.near_score <= max_frac * rep.branches + 2, f"near-threshold branches: {rep.summary()}"
    assert rep.near_route_diff <= 1e-3 * rep.tokens_routed + 1, f"excluded tokens that differ: {rep.summary()}"
    assert rep.near_score_diff <= 1e-3 * rep.branches + 1, f"excluded branches that differ: {rep.summary()}"


def check_adaln(rep: Report, cfg, w: dict, pre: dict | None, post: dict, tr: dict, refresh: bool, cond,
                tol: float = 1e-2):
    """Teacher-forced check of an AdaLN block's modulation and attention
    sub-layer (Sec. 3 residual form under the Sec. 4.1 cache).  Returns
    (router input, residual u, gate_m token rows) for the MoE check; the
    trace's layer_in is the MoE input m."""
    wo = oracle_weights(w)
    D = cfg.hidden
    x = np_of(tr["block_in"]).astype(np.float64)
    T = x.shape[0]
    S = cfg.seq_len or T
    eps = float(np.float32(cfg.ln_eps))
    # ---- modulation: float32 dot products of D terms against the float64 oracle
    c = np.asarray(cond, np.float64)
    mod_g = np_of(tr["mod"]).astype(np.float64).reshape(T // S, 6, D)
    mod_o = O.adaln_modulation(c, wo["w_ada"], wo.get("b_ada"))
    mag = (np.abs(O.silu(c)) @ np.abs(wo["w_ada"]).T).reshape(T // S, 6, D)
    err = np.abs(mod_g - mod_o)
    assert (err <= 1e-5 * mag + 1e-6).all(), f"modulation: worst err {err.max():.3e}"
    rows6 = [O.token_rows(mod_g[:, j], T, S) for j in range(6)]
    # ---- attention from h = LN-modulate(x)
    h = O.round_bf16(O.modulate(O.layer_norm(x, eps), rows6[0], rows6[1]))
    a_post = np_of(post["attn_a"]).astype(np.float64)
    full = refresh or cfg.attn_policy == 2
    has_pre = pre is not None and pre["n_tokens"]
    a_pre = np_of(pre["attn_a"]).astype(np.float64) if has_pre else None
    if full:
        rows = np.arange(T)
    elif cfg.attn_policy == 1:
        rows = np.zeros(0, np.int64)
    else:
        rows = np.nonzero(np_of(tr["token_any"]))[0]
    if len(rows):
        a_o = O.attention(h, wo["w_qkv"], wo.get("b_qkv"), wo["w_o"], wo.get("b_o"), cfg.n_heads, cfg.seq_len, rows)
        rl = rel_l2(a_post[rows], a_o)
        rep.max_attn_rel_l2 = max(rep.max_attn_rel_l2, rl)
        assert rl <= tol, f"attention rows rel L2 {rl:.3e}"
        per_row = np.linalg.norm(a_post[rows] - a_o, axis=1) / np.maximum(np.linalg.norm(a_o, axis=1), 1e-30)
        assert per_row.max() <= 4 * tol, f"worst attention row rel L2 {per_row.max():.3e}"
    kept = np.setdiff1d(np.arange(T), rows)
    if len(kept):
        assert a_pre is not None, "a cache step without a cached attention output"
        assert np.array_equal(a_post[kept], a_pre[kept]), "kept attention rows changed"
    # ---- residual u = x + g_a a and MoE input m = LN-modulate(u), from the GPU's a and u
    u = np_of(tr["resid"]).astype(np.float64)
    m = np_of(tr["layer_in"]).astype(np.float64)
    close_in_bf16(u, x + rows6[2] * a_post, "residual u", floor=2.0 ** -22 * (np.abs(x) + np.abs(rows6[2] * a_post)))

    def ln_floor(v):
        # float32 mean / rsqrt over D and the two products: 1e-5 of the terms
        return 1e-5 * (np.abs(O.layer_norm(v, eps) * (1 + rows6[4])) + np.abs(rows6[3]))

    close_in_bf16(m, O.modulate(O.layer_norm(u, eps), rows6[3], rows6[4]), "MoE input m", floor=ln_floor(u))
    r = np_of(tr["route_in"]).astype(np.float64)
    if full or cfg.attn_policy == 1:
        assert np.array_equal(r, m), "router input differs from the MoE input"
    else:
        u_pre = O.round_bf16(x + rows6[2] * a_pre)
        close_in_bf16(r, O.modulate(O.layer_norm(u_pre, eps), rows6[3], rows6[4]), "router input m'",
                      floor=ln_floor(u_pre))
        assert np.array_equal(r[kept], m[kept]), "kept tokens' MoE input differs from their router input"
    rep.attn_rows += len(rows)
    return r, u, rows6[5]


def check_layer(rep: Report, cfg, w: dict, pre: dict | None, post: dict, tr: dict, out_gpu: np.ndarray,
                refresh: bool, bf16: bool, out_tol=None, route_in=None, resid=None, gate=None):
    """Teacher-forced comparison of one layer step.  Raises AssertionError.

    ``route_in`` is the router input when it differs from the FFN input
    (a DiT-MoE block on a sync cache step)."""
    T = tr["route_e"].shape[0]
    D, E, k, S = cfg.hidden, cfg.n_experts, cfg.top_k, cfg.n_shared
    prm = params_of(cfg)
    wo = oracle_weights(w)
    u = np_of(tr["layer_in"]).astype(np.float64)
    u_route = u if route_in is None else np.asarray(route_in, np.float64)
    e_g = np_of(tr["route_e"]).astype(np.int64)
    w_g = np_of(tr["route_w"]).astype(np.float64)
    # ---- router (Eq. 7)
    e_o, w_o, ok, cond = count_route_margins(rep, u_route, wo, k, prm.renorm_topk, e_g)
    bad = np.nonzero(ok & (e_o != e_g).any(axis=1))[0]
    assert len(bad) == 0, f"top-k ids differ on {len(bad)} tokens, e.g. {bad[:5]}: gpu {e_g[bad[:3]]} oracle {e_o[bad[:3]]}"
    check_gate_weights(w_g[ok], w_o[ok], cond[ok])
    # ---- EMA (Eq. 10) from the GPU's pre-step statistic and routing
    C_pre = np.zeros((E, T)) if (pre is None or pre["n_tokens"] == 0) else np_of(pre["ema"]).astype(np.float64).T
    C_o = O.ema_update(C_pre, e_g, prm.beta)
    C_g = np_of(post["ema"]).astype(np.float64).T
    assert np.allclose(C_g, C_o, rtol=2e-6, atol=1e-7), f"EMA: max err {np.abs(C_g - C_o).max()}"
    # ---- tau (Eq. 11-12) from the GPU's statistic
    tau_o = O.expert_threshold(O.normalized_entropy(C_g, prm.entropy_norm), prm.tau0, prm.alpha)
    tau_g = np_of(tr["tau"]).astype(np.float64)
    fin = np.isfinite(tau_o)
    assert np.allclose(tau_g[fin], tau_o[fin], rtol=1e-5, atol=1e-6), f"tau: {tau_g} vs {tau_o}"
    assert np.array_equal(np.isinf(tau_g), np.isinf(tau_o))
    # ---- select (Sec. 4.2, Eq. 9) from the GPU routing, tau and pre-step cache
    st_pre = state_to_oracle(pre, T, D, E, k, S)
    sel = O.select_branches(e_g, w_g, st_pre.cache_e, st_pre.cache_w, st_pre.cache_norm, tau_g,
                            prm.lambda1, prm.lambda2, refresh, prm.score_terms, prm.granularity)
    rec_g = np_of(tr["recompute"]).astype(bool)
    slot_g = np_of(tr["slot"]).astype(np.int64)
    mat_g = np_of(tr["matched"]).astype(bool)
    assert np.array_equal(slot_g, sel["slot"]), "slots differ"
    assert np.array_equal(mat_g, sel["matched"]), "matched flags differ"
    far = sel["margin"] >= NEAR
    rep.near_score += int((~far).sum())
    rep.near_score_diff += int((~far & (rec_g != sel["recompute"])).sum())
    diff = far & (rec_g != sel["recompute"])
    assert not diff.any(), f"recompute mask differs on {int(diff.sum())} branches"
    any_g = np_of(tr["token_any"]).astype(bool)
    assert np.array_equal(any_g, rec_g.any(axis=1))
    # ---- compaction
    cnt, off, flat = expected_lists(e_g, rec_g, slot_g, any_g, E, k, S, refresh, cfg.shared_policy == 1)
    assert np.array_equal(np_of(tr["counts"]), cnt), "group counts"
    assert np.array_equal(np_of(tr["offsets"]), off), "group offsets"
    assert np.array_equal(np_of(tr["list"])[: off[-1]], flat), "row lists"
    # ---- FFN + combine (Eq. 5, Eq. 8) from the GPU decisions and pre-step cache
    out_o, new_o, _ = O.recompute_and_combine(st_pre, u, e_g, w_g, rec_g, slot_g, wo, prm, refresh,
                                              resid=resid, gate=gate)
    # A few wrong rows can hide under a global bound: every token row too.
    shared_rows = (np.ones(T, bool) if refresh or cfg.shared_policy == 1 else rec_g.any(axis=1)) if S else None
    terms = fresh_terms(u, wo, e_g, w_g, rec_g, slot_g, new_o, prm.gelu, gate, shared_rows) if bf16 else None
    check_output(rep, out_gpu, out_o, bf16, out_tol if out_tol is not None else (1e-2 if bf16 else 1e-5),
                 terms=terms)
    ch_g = np_of(post["cache_h"]).astype(np.float64)
    fresh = np.zeros((T, k), bool)
    for i, p in np.argwhere(rec_g):
        fresh[i, slot_g[i, p]] = True
    if fresh.any():
        tol_h = 1e-2 if bf16 else 1e-5
        rf = rel_l2(ch_g[fresh], new_o.cache_h[fresh])
        assert rf <= tol_h, f"fresh cache rows rel L2 {rf:.3e}"
        per = (np.linalg.norm(ch_g[fresh] - new_o.cache_h[fresh], axis=1)
               / np.maximum(np.linalg.norm(new_o.cache_h[fresh], axis=1), 1e-30))
        assert per.max() <= 4 * tol_h, f"worst fresh cache row rel L2 {per.max():.3e}"
    if (~fresh).any() and pre is not None and pre["n_tokens"]:
        assert np.array_equal(ch_g[~fresh], st_pre.cache_h[~fresh]), "reused cache rows changed"
    assert np.array_equal(np_of(post["cache_e"]), new_o.cache_e), "cache expert ids"
    assert np.array_equal(np_of(post["cache_w"]).astype(np.float64), new_o.cache_w.astype(np.float32).astype(np.float64)), "cache weights"
    nrm = np.sqrt((ch_g ** 2).sum(axis=2))
    assert np.allclose(np_of(post["cache_norm"]), nrm, rtol=2e-5, atol=1e-6), "cached norms"
    if S:
        sh_g = np_of(post["shared_h"]).astype(np.float64)
        rs = rel_l2(sh_g, new_o.shared_h)
        assert rs <= (1e-2 if bf16 else 1e-5), f"shared rows rel L2 {rs:.3e}"
    if cfg.token_reuse_policy:
        # Sec. 4.1 token level: tokens with an empty recompute set keep y^{t0}
        # bit for bit; the others store their new y.
        y_g = np_of(post["cache_y"]).astype(np.float64)
        keep = ~any_g if not refresh else np.zeros(T, bool)
        if keep.any():
            assert np.array_equal(y_g[keep], st_pre.cache_y[keep]), "a reused token's y changed"
            rep.tokens_copied += int(keep.sum())
        if (~keep).any():
            ry = rel_l2(y_g[~keep], new_o.cache_y[~keep])
            assert ry <= (1e-2 if bf16 else 1e-5), f"stored y rel L2 {ry:.3e}"
    rep.layers_checked += 1
    rep.branches += T * k
    rep.recomputed += int(rec_g.sum())
    rep.reused += int((~rec_g).sum())
    rep.unmatched += int((~mat_g).sum()) if not refresh else 0


def run_trajectory(stack, cfg, layer_weights, xs, refresh_flags=None, check=True, bf16=True, out_tol=None,
                   forces=None, conds=None, next_input=None, n_steps=None):
    """Step the GPU stack over ``xs`` and check every layer of every step
    (``conds[t]``: the per-sample conditioning of an AdaLN stack).  With
    ``next_input``, xs[0] starts ``n_steps`` steps and step t > 0 takes
    next_input(t, previous output)."""
    import torch
    rep = Report()
    dt = torch.bfloat16 if bf16 else torch.float32
    L = cfg.n_layers
    prev_T = None
    n = len(xs) if next_input is None else n_steps
    out = None
    for t in range(n):
        # A sampler loop feeds each step's output through ``next_input``.
        x = xs[t] if next_input is None or t == 0 else next_input(t, out)
        T = x.shape[0]
        force = bool(forces and forces[t])
        N = cfg.refresh_period
        refresh = force or prev_T != T or t == 0 or (N > 0 and t % N == 0)
        if refresh_flags is not None:
            refresh_flags.append(refresh)
        pre = [stack.get_state(l) for l in range(L)] if check else None
        if check and prev_T != T:
            pre = [None] * L
        xd = torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda().to(dt)
        cd = None if conds is None else torch.from_numpy(np.ascontiguousarray(conds[t], np.float32)).cuda()
        out = stack.step(xd, t, force_refresh=force, cond=cd)
        torch.cuda.synchronize()
        if check:
            block = cfg.n_heads > 0
            for l in range(L):
                tr = stack.get_trace(l, T)
                post = stack.get_state(l)
                if l + 1 < L:
                    out_l = np_of(stack.get_trace(l + 1, T)["block_in" if block else "layer_in"]).astype(np.float64)
                else:
                    out_l = np_of(out).astype(np.float64)
                resid = gate = None
                if cfg.adaln:
                    route_in, resid, gate = check_adaln(rep, cfg, layer_weights[l], pre[l], post, tr, refresh,
                                                        conds[t])
                elif block:
                    route_in = check_attention(rep, cfg, layer_weights[l], pre[l], post, tr, refresh)
                else:
                    route_in = None
                check_layer(rep, cfg, layer_weights[l], pre[l], post, tr, out_l, refresh, bf16, out_tol,
                            route_in=route_in, resid=resid, gate=gate)
        rep.steps += 1
        prev_T = T
    if check:
        st = stack.stats()
        rep.lib_near_route, rep.lib_near_score = st["near_margin_route"], st["near_margin_score"]
        REPORTS.append((os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0], rep))
        assert_margins(rep)
    return rep, out
