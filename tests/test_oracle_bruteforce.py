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
]


def _bf_params(prm: O.Params) -> dict:
    return dict(top_k=prm.top_k, lambda1=prm.lambda1, lambda2=prm.lambda2, tau0=prm.tau0,
                alpha=prm.alpha, beta=prm.beta, renorm_topk=prm.renorm_topk,
                entropy_norm=prm.entropy_norm, shared_policy=prm.shared_policy,
                reused_meta_policy=prm.reused_meta_policy, gelu=prm.gelu, score_terms=prm.score_terms,
                granularity=prm.granularity)


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
        if not refresh:
            kinds |= {("reuse", bool(b)) for b in (~inf["recompute"]).ravel()}
            kinds |= {("unmatched", bool(b)) for b in (~inf["matched"]).ravel()}
    if T > 1 and k < E:
        assert ("reuse", True) in kinds and ("unmatched", True) in kinds, kinds
