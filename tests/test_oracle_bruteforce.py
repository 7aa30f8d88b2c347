"""Oracle vs the pure-Python brute force on tiny cases (T <= 8, E <= 4).

Multi-step trajectories with a mix of matched, unmatched, reused and
recomputed branches; every switch of the readings is exercised once.
"""
import math

import numpy as np
import pytest

import bruteforce_ref as BF
from oracle import moeca_oracle as O
from paper_2606_15615_gb300.workloads import tiny_layer

CASES = [
    # (seed, T, D, E, k, F, n_shared, bias, overrides)
    (1, 8, 6, 4, 2, 5, 0, False, {}),
    (2, 7, 5, 4, 3, 4, 0, True, {}),
    (3, 8, 4, 3, 1, 3, 1, False, {"tau0": 1.4}),
    (4, 6, 6, 4, 2, 4, 1, True, {"shared_policy": "always"}),
    (5, 8, 5, 4, 2, 6, 0, False, {"entropy_norm": "minmax"}),
    (6, 8, 4, 4, 2, 3, 0, False, {"reused_meta_policy": "overwrite"}),
    (7, 5, 4, 4, 4, 3, 0, False, {"gelu": "erf"}),
    (8, 8, 6, 4, 2, 5, 0, False, {"renorm_topk": False, "tau0": 0.5}),
    (9, 1, 4, 3, 2, 3, 0, False, {}),
    # Table 5's score-signal subsets and token-level granularity (Sec. 3)
    (10, 8, 6, 4, 2, 5, 0, False, {"score_terms": 1, "tau0": 0.55}),
    (11, 8, 6, 4, 2, 5, 0, False, {"score_terms": 2, "tau0": 0.08}),
    (18, 8, 6, 4, 2, 5, 0, False, {"score_terms": 4, "tau0": 0.25}),
    (13, 8, 6, 4, 2, 5, 0, False, {"score_terms": 3, "tau0": 0.6}),
    (14, 8, 6, 4, 2, 5, 0, False, {"score_terms": 5, "tau0": 0.75}),
    (15, 8, 6, 4, 2, 5, 0, False, {"score_terms": 6, "tau0": 0.3}),
    (16, 8, 6, 4, 2, 5, 1, False, {"granularity": "token", "tau0": 1.1}),
    (17, 8, 5, 4, 3, 4, 0, True, {"granularity": "token", "score_terms": 3, "tau0": 0.9}),
    # Sec. 4.1's "reuse cached states" reading: R_i empty => y_i^{t0} copied
    (19, 8, 6, 4, 2, 5, 0, False, {"token_reuse_policy": "copy", "tau0": 1.1}),
    (20, 8, 5, 4, 2, 4, 1, True, {"token_reuse_policy": "copy", "tau0": 1.3}),
    (21, 8, 6, 4, 2, 5, 0, False, {"token_reuse_policy": "copy", "granularity": "token", "tau0": 1.2}),
]


def _bf_params(prm: O.Params) -> dict:
    return dict(top_k=prm.top_k, lambda1=prm.lambda1, lambda2=prm.lambda2, tau0=prm.tau0,
                alpha=prm.alpha, beta=prm.beta, renorm_topk=prm.renorm_topk,
                entropy_norm=prm.entropy_norm, shared_policy=prm.shared_policy,
                reused_meta_policy=prm.reused_meta_policy, gelu=prm.gelu, score_terms=prm.score_terms,
                granularity=prm.granularity, token_reuse_policy=prm.token_reuse_policy)


@pytest.mark.parametrize("case", CASES, ids=[f"case{c[0]}" for c in CASES])
def test_oracle_equals_bruteforce(case):
    seed, T, D, E, k, F, S, bias, over = case
    w, x0, rng = tiny_layer(seed, T, D, E, k, F, n_shared=S, bias=bias, wscale=0.6)
    prm = O.Params(top_k=k, tau0=over.pop("tau0", 0.8), refresh_period=4, **over)
    st = O.Stack([w], prm, D, E, S)
    bstate = BF.empty_state(T, D, E, k, S)
    kinds = set()
    x = x0
    for t in range(7):
        if t:
            x = (x + 0.35 * rng.standard_normal(x.shape)).astype(np.float32)
        refresh = st.is_refresh(t, T)
        out, infos = st.step(x, t)
        inf = infos[0]
        bout, bstate, dec = BF.layer_step(bstate, x.tolist(), {kk: (None if v is None else v.tolist())
                                                               for kk, v in w.items()},
                                          _bf_params(prm), refresh)
        assert inf["e"].tolist() == dec["e"]
        np.testing.assert_allclose(inf["w"], dec["w"], rtol=1e-12)
        np.testing.assert_allclose(inf["tau"], dec["tau"], rtol=1e-12)
        assert inf["recompute"].tolist() == dec["recompute"]
        assert inf["slot"].tolist() == dec["slot"]
        np.testing.assert_allclose(out, bout, rtol=1e-11, atol=1e-12)
        s = st.states[0]
        np.testing.assert_allclose(s.C, bstate["C"], rtol=1e-12)
        assert s.cache_e.tolist() == bstate["cache_e"]
        np.testing.assert_allclose(s.cache_w, bstate["cache_w"], rtol=1e-12)
        np.testing.assert_allclose(s.cache_norm, bstate["cache_norm"], rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(s.cache_h, bstate["cache_h"], rtol=1e-11, atol=1e-13)
        if S:
            np.testing.assert_allclose(s.shared_h, bstate["shared_h"], rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(s.cache_y, bstate["cache_y"], rtol=1e-11, atol=1e-13)
        if not refresh:
            kinds |= {("reuse", bool(b)) for b in (~inf["recompute"]).ravel()}
            kinds |= {("unmatched", bool(b)) for b in (~inf["matched"]).ravel()}
            kinds |= {("token_reused", bool(b)) for b in (~inf["recompute"].any(axis=1))}
    if T > 1 and k < E:
        assert ("reuse", True) in kinds and ("unmatched", True) in kinds, kinds
    if prm.token_reuse_policy == "copy":
        assert ("token_reused", True) in kinds and ("token_reused", False) in kinds, kinds


ADALN_CASES = [
    # (seed, T, S, D, H, E, k, F, n_shared, policy, tau0)
    (31, 8, 4, 8, 2, 4, 2, 5, 0, "sync", 0.75),
    (32, 8, 4, 8, 2, 4, 2, 5, 1, "sync", 0.9),
    (33, 6, 3, 6, 3, 3, 1, 4, 0, "stale", 1.4),  # k = 1: a matched score is 1 + lambda2
    (34, 8, 8, 8, 2, 4, 2, 5, 0, "full", 0.75),
    (35, 8, 4, 8, 2, 4, 2, 5, 1, "sync", 1.2, "copy"),  # Sec. 4.1 "reuse cached states" reading
]


@pytest.mark.parametrize("case", ADALN_CASES, ids=[f"adaln{c[0]}" for c in ADALN_CASES])
def test_adaln_block_equals_bruteforce(case):
    """The oracle's AdaLN block (Sec. 3 residual form under the Sec. 4.1 cache)
    against scalar loops: modulation, layer norm, per-head attention, the
    sync rule's attention update and the gated combine, over 6 steps with the
    conditioning changing every step."""
    from paper_2606_15615_gb300.workloads import conditioning, tiny_adaln, tiny_attn
    seed, T, S, D, H, E, k, F, n_sh, policy, tau0 = case[:11]
    reuse = case[11] if len(case) > 11 else "current"
    w, x0, rng = tiny_layer(seed, T, D, E, k, F, n_shared=n_sh, bias=True, wscale=0.6)
    w.update(tiny_attn(seed, D, wscale=0.5))
    w.update(tiny_adaln(seed, D, wscale=0.4))
    prm = O.Params(top_k=k, tau0=tau0, refresh_period=4, n_heads=H, seq_len=S, attn_policy=policy, adaln=True,
                   token_reuse_policy=reuse)
    st = O.Stack([w], prm, D, E, n_sh)
    bprm = dict(_bf_params(prm), n_heads=H, seq_len=S, attn_policy=policy, ln_eps=prm.ln_eps)
    bstate = BF.empty_state(T, D, E, k, n_sh)
    bstate["attn_a"] = [[0.0] * D for _ in range(T)]
    conds = conditioning(seed, T // S, D, 6)
    wl = {kk: (None if v is None else v.tolist()) for kk, v in w.items()}
    kinds = set()
    x = x0
    for t in range(6):
        if t:
            x = (x + 0.3 * rng.standard_normal(x.shape)).astype(np.float32)
        refresh = st.is_refresh(t, T)
        out, infos = st.step(x, t, cond=conds[t])
        inf = infos[0]
        bout, bstate, dec = BF.adaln_block_step(bstate, x.tolist(), conds[t].tolist(), wl, bprm, refresh)
        assert inf["e"].tolist() == dec["e"]
        assert inf["recompute"].tolist() == dec["recompute"]
        assert inf["slot"].tolist() == dec["slot"]
        assert sorted(inf["attn_rows"].tolist()) == sorted(dec["attn_rows"])
        np.testing.assert_allclose(inf["u"], dec["u"], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(inf["m"], dec["m"], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(out, bout, rtol=1e-10, atol=1e-11)
        s = st.states[0]
        np.testing.assert_allclose(s.attn_a, bstate["attn_a"], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(s.cache_h, bstate["cache_h"], rtol=1e-10, atol=1e-12)
        if not refresh:
            kinds |= {("reuse", bool(b)) for b in (~inf["recompute"]).ravel()}
            if policy == "sync":
                kinds.add(("partial_attention", 0 < len(dec["attn_rows"]) < T))
            kinds |= {("token_reused", not any(r)) for r in dec["recompute"]}
    assert ("reuse", True) in kinds and ("reuse", False) in kinds, kinds
    if reuse == "copy":
        assert ("token_reused", True) in kinds, kinds
    if policy == "sync":
        assert ("partial_attention", True) in kinds, kinds
