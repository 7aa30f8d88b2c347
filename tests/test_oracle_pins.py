"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a closed form,
a special case, an invariant of the definitions, a textbook formulation written
independently (dense einsum MoE), or exact reuse.  The brute-force and
hand-worked fixture pins live in their own files.
"""
import math

import numpy as np
import pytest

from oracle import moeca_oracle as O
from paper_2606_15615_gb300.workloads import tiny_layer


def _softmax_rows(z):
    z = z - z.max(axis=1, keepdims=True)
    ez = np.exp(z)
    return ez / ez.sum(axis=1, keepdims=True)


def _gelu_tanh(z):
    return 0.5 * z * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (z + 0.044715 * z ** 3)))


def textbook_moe(u, w, k):
    """Eq. 5 / Eq. 6 as a dense computation: every expert on every token, then gated.

    Independent of the oracle: einsum over all experts, top-k by lexsort.
    """
    u = u.astype(np.float64)
    z = np.einsum("td,ed->te", u, w["w_gate"].astype(np.float64))
    if w.get("b_gate") is not None:
        z = z + w["b_gate"][None, :]
    T, E = z.shape
    z32 = z.astype(np.float32)
    gate = np.zeros((T, E))
    probs = _softmax_rows(z)
    for t in range(T):
        order = np.lexsort((np.arange(E), -z32[t]))[:k]
        g = probs[t, order] / probs[t, order].sum()
        gate[t, order] = g
    hid = _gelu_tanh(np.einsum("td,efd->tef", u, w["w1"].astype(np.float64)))
    outs = np.einsum("tef,edf->ted", hid, w["w2"].astype(np.float64))
    y = np.einsum("te,ted->td", gate, outs)
    if w.get("ws1") is not None:
        hs = _gelu_tanh(np.einsum("td,sfd->tsf", u, w["ws1"].astype(np.float64)))
        y = y + np.einsum("tsf,sdf->td", hs, w["ws2"].astype(np.float64))
    return u + y


# --- Routing (Eq. 7) --------------------------------------------------------

def test_topk_weights_renormalised_sum_to_one():
    w, x, _ = tiny_layer(1, T=64, D=16, E=8, k=3, F=8, bias=True)
    e, wt, _, _ = O.route(x, w["w_gate"], w["b_gate"], 3, renorm=True)
    np.testing.assert_allclose(wt.sum(axis=1), 1.0, rtol=0, atol=1e-12)
    assert (wt[:, :-1] >= wt[:, 1:] - 1e-15).all(), "branches are ordered by descending weight"
    for row in e:
        assert len(set(row.tolist())) == 3


def test_topk_without_renorm_keeps_softmax_ratios():
    # Softmax fixes w_p / w_p' = exp(z_p - z_p') and sum over all E of p = 1.
    w, x, _ = tiny_layer(2, T=32, D=12, E=6, k=2, F=4)
    e, wt, _, _ = O.route(x, w["w_gate"], None, 2, renorm=False)
    z = x.astype(np.float64) @ w["w_gate"].astype(np.float64).T
    for t in range(32):
        np.testing.assert_allclose(wt[t, 0] / wt[t, 1], math.exp(z[t, e[t, 0]] - z[t, e[t, 1]]), rtol=1e-12)
        assert wt[t].sum() < 1.0
    np.testing.assert_allclose(O.route(x, w["w_gate"], None, 6, renorm=False)[1].sum(axis=1), 1.0, atol=1e-12)


def test_topk_ties_go_to_lower_expert_id():
    wg = np.array([[1.0, 0.0], [1.0, 0.0], [0.5, 0.0], [1.0, 0.0]])
    e, wt, near, _ = O.route(np.array([[2.0, 1.0]]), wg, None, 2, renorm=True)
    assert e.tolist() == [[0, 1]]
    np.testing.assert_allclose(wt, [[0.5, 0.5]])
    assert near[0] == 0.0


# --- EMA, entropy, threshold (Eq. 10-12) ------------------------------------

@pytest.mark.parametrize("beta", [0.45, 0.65, 0.85])
def test_ema_closed_form(beta):
    # Routed for n steps from C = 0: C = 1 - beta^n; then unrouted m steps: times beta^m.
    C = np.zeros((2, 1))
    for n in range(1, 9):
        C = O.ema_update(C, np.array([[0]]), beta)
        assert C[0, 0] == pytest.approx(1.0 - beta ** n, rel=1e-12)
        assert C[1, 0] == 0.0
    for m in range(1, 5):
        C = O.ema_update(C, np.array([[1]]), beta)
        assert C[0, 0] == pytest.approx((1.0 - beta ** 8) * beta ** m, rel=1e-12)
        assert C[1, 0] == pytest.approx(1.0 - beta ** m, rel=1e-12)


def test_threshold_special_cases():
    T = 16
    uniform = np.full((1, T), 0.3)
    onehot = np.zeros((1, T)); onehot[0, 5] = 0.9
    rng = np.random.default_rng(0)
    rand = rng.random((3, T))
    for tau0, alpha in [(0.8, 0.6), (0.65, 0.3), (1.0, 0.9)]:
        assert O.expert_threshold(O.normalized_entropy(uniform), tau0, alpha)[0] == pytest.approx(tau0 * (1 + alpha))
        assert O.expert_threshold(O.normalized_entropy(onehot), tau0, alpha)[0] == pytest.approx(tau0 * (1 - alpha))
        np.testing.assert_allclose(O.expert_threshold(O.normalized_entropy(rand), tau0, 0.0), tau0)
    Hbar = O.normalized_entropy(rand)
    assert ((Hbar > 0) & (Hbar < 1)).all()


def test_entropy_two_point_and_scale_invariance():
    # Mass split evenly over m positions gives H = ln m, whatever the scale of C.
    for m in (1, 2, 3, 7):
        C = np.zeros((1, 10)); C[0, :m] = 0.123
        assert O.spatial_entropy(C)[0] == pytest.approx(math.log(m), abs=1e-12)
        assert O.spatial_entropy(5.0 * C)[0] == pytest.approx(math.log(m), abs=1e-12)


def test_entropy_minmax_mode():
    C = np.array([[1.0, 0, 0, 0], [1.0, 1.0, 0, 0], [1.0, 1.0, 1.0, 1.0], [0, 0, 0, 0]])
    np.testing.assert_allclose(O.normalized_entropy(C, "minmax"), [0.0, 0.5, 1.0, 0.5])


# --- Scoring and selection (Eq. 9) ------------------------------------------

def test_historical_contribution_sums_to_one():
    n = np.abs(np.random.default_rng(3).standard_normal((50, 4)))
    n[7] = 0.0
    o = O.historical_contribution(n)
    np.testing.assert_allclose(np.delete(o, 7, axis=0).sum(axis=1), 1.0, atol=1e-12)
    assert (o[7] == 0).all()


def _run(layer_w, prm, xs, n_shared=0):
    D = xs[0].shape[1]
    E = layer_w["w_gate"].shape[0]
    st = O.Stack([layer_w], prm, D, E, n_shared)
    outs, infos = [], []
    for t, x in enumerate(xs):
        o, inf = st.step(x, t)
        outs.append(o)
        infos.append(inf[0])
    return outs, infos, st


def test_identical_input_matches_every_branch_with_zero_drift():
    w, x, _ = tiny_layer(4, T=40, D=16, E=6, k=2, F=8)
    prm = O.Params(top_k=2, tau0=0.8)
    st = O.Stack([w], prm, 16, 6)
    st.step(x, 0)
    norms_before = st.states[0].cache_norm.copy()
    _, infos = st.step(x, 1)
    inf = infos[0]
    assert inf["matched"].all()
    o = O.historical_contribution(norms_before)[np.arange(40)[:, None], inf["slot"]]
    # Same routing, so Delta = 0 and s = w + lambda2 * o.
    np.testing.assert_allclose(inf["score"], inf["w"] + prm.lambda2 * o, rtol=1e-12)


def test_reuse_disabled_equals_textbook_moe():
    # tau0 = -inf recomputes every branch on every step: Eq. 5 at each step.
    w, x0, rng = tiny_layer(5, T=48, D=16, E=5, k=2, F=12, bias=True)
    prm = O.Params(top_k=2, tau0=-math.inf)
    xs = [x0 + 0.1 * t * rng.standard_normal(x0.shape).astype(np.float32) for t in range(4)]
    outs, infos, _ = _run(w, prm, xs)
    for x, o, inf in zip(xs, outs, infos):
        assert inf["recompute"].all()
        np.testing.assert_allclose(o, textbook_moe(x, w, 2), rtol=1e-12, atol=1e-12)


def test_reuse_disabled_with_shared_expert_equals_textbook_moe():
    w, x0, rng = tiny_layer(6, T=32, D=8, E=4, k=2, F=6, n_shared=1)
    prm = O.Params(top_k=2, tau0=-math.inf)
    xs = [x0, x0 + 0.2 * rng.standard_normal(x0.shape).astype(np.float32)]
    outs, _, _ = _run(w, prm, xs, n_shared=1)
    for x, o in zip(xs, outs):
        np.testing.assert_allclose(o, textbook_moe(x, w, 2), rtol=1e-12, atol=1e-12)


def test_refresh_every_step_equals_textbook_moe():
    w, x0, rng = tiny_layer(7, T=32, D=8, E=4, k=2, F=6)
    prm = O.Params(top_k=2, tau0=10.0, refresh_period=1)
    xs = [x0 + 0.3 * t * rng.standard_normal(x0.shape).astype(np.float32) for t in range(3)]
    outs, infos, _ = _run(w, prm, xs)
    for x, o, inf in zip(xs, outs, infos):
        assert inf["refresh"]
        np.testing.assert_allclose(o, textbook_moe(x, w, 2), rtol=1e-12, atol=1e-12)


def test_everything_reused_returns_cached_output_exactly():
    w, x, _ = tiny_layer(8, T=40, D=16, E=6, k=3, F=8, n_shared=1)
    prm = O.Params(top_k=3, tau0=math.inf)
    outs, infos, _ = _run(w, prm, [x, x, x], n_shared=1)
    assert not infos[1]["recompute"].any() and not infos[2]["recompute"].any()
    assert np.array_equal(outs[1], outs[0]) and np.array_equal(outs[2], outs[0])


def test_slots_are_a_permutation_and_cache_holds_current_experts():
    w, x0, rng = tiny_layer(9, T=64, D=16, E=8, k=3, F=8)
    prm = O.Params(top_k=3, tau0=0.9)
    xs = [x0 + 0.5 * t * rng.standard_normal(x0.shape).astype(np.float32) for t in range(5)]
    outs, infos, st = _run(w, prm, xs)
    saw_unmatched = saw_reuse = False
    for inf in infos:
        for i in range(64):
            assert sorted(inf["slot"][i].tolist()) == [0, 1, 2]
        saw_unmatched |= bool((~inf["matched"] & ~np.array(inf["refresh"])).any())
        saw_reuse |= bool((~inf["recompute"]).any())
    assert saw_unmatched and saw_reuse
    last = infos[-1]
    state = st.states[0]
    for i in range(64):
        for p in range(3):
            assert state.cache_e[i, last["slot"][i, p]] == last["e"][i, p]


def test_recomputed_branch_equals_fresh_ffn_and_reused_keeps_old_weight():
    w, x0, rng = tiny_layer(10, T=64, D=16, E=6, k=2, F=8)
    prm = O.Params(top_k=2, tau0=0.75)
    xs = [x0, x0 + 0.05 * rng.standard_normal(x0.shape).astype(np.float32)]
    outs, infos, st = _run(w, prm, xs)
    inf, state = infos[1], st.states[0]
    rec = inf["recompute"]
    assert rec.any() and (~rec).any()
    for i, p in np.argwhere(rec):
        e = inf["e"][i, p]
        h = O.gelu(xs[1][i].astype(np.float64) @ w["w1"][e].T.astype(np.float64)) @ w["w2"][e].T.astype(np.float64)
        np.testing.assert_allclose(state.cache_h[i, inf["slot"][i, p]], h, rtol=1e-12)
        assert state.cache_w[i, inf["slot"][i, p]] == inf["w"][i, p]
    for i, p in np.argwhere(~rec):
        q = inf["slot"][i, p]
        assert state.cache_w[i, q] == infos[0]["w"][i, q]  # kept w^{t0}


def test_shared_expert_follows_synchronized_rule():
    w, x0, rng = tiny_layer(11, T=64, D=8, E=4, k=2, F=6, n_shared=1)
    prm = O.Params(top_k=2, tau0=0.9)
    x1 = x0 + 0.05 * rng.standard_normal(x0.shape).astype(np.float32)
    outs, infos, st = _run(w, prm, [x0, x1], n_shared=1)
    any1 = infos[1]["token_any"]
    assert any1.any() and (~any1).any()
    fresh = O.expert_ffn(x1.astype(np.float64), w["ws1"][0], w["ws2"][0], "tanh")
    old = O.expert_ffn(x0.astype(np.float64), w["ws1"][0], w["ws2"][0], "tanh")
    np.testing.assert_allclose(st.states[0].shared_h[any1], fresh[any1], rtol=1e-12)
    np.testing.assert_allclose(st.states[0].shared_h[~any1], old[~any1], rtol=1e-12)


def test_reused_meta_overwrite_policy():
    w, x0, rng = tiny_layer(12, T=48, D=8, E=4, k=2, F=6)
    prm = O.Params(top_k=2, tau0=0.9, reused_meta_policy="overwrite")
    x1 = x0 + 0.05 * rng.standard_normal(x0.shape).astype(np.float32)
    _, infos, st = _run(w, prm, [x0, x1])
    inf = infos[1]
    for i, p in np.argwhere(~inf["recompute"]):
        assert st.states[0].cache_w[i, inf["slot"][i, p]] == inf["w"][i, p]


def test_refresh_schedule():
    w, x, _ = tiny_layer(13, T=8, D=8, E=4, k=2, F=4)
    st = O.Stack([w], O.Params(top_k=2, refresh_period=3), 8, 4)
    flags = [st.step(x, t)[1][0]["refresh"] for t in range(7)]
    assert flags == [True, False, False, True, False, False, True]
    assert st.step(x[:5], 7)[1][0]["refresh"], "a new token count forces a full step"
    assert st.step(x[:5], 8, force=True)[1][0]["refresh"]


def _random_selection_inputs(seed, T=64, k=3, E=6):
    rng = np.random.default_rng(seed)
    e_cur = np.stack([rng.permutation(E)[:k] for _ in range(T)])
    w_cur = rng.dirichlet(np.ones(k), size=T)
    # Caches that share some experts with the current routing.
    cache_e = np.stack([rng.permutation(E)[:k] for _ in range(T)])
    cache_e[: T // 2] = e_cur[: T // 2][:, rng.permutation(k)]
    cache_w = rng.dirichlet(np.ones(k), size=T)
    cache_norm = rng.uniform(0.1, 2.0, size=(T, k))
    tau = rng.uniform(0.3, 0.9, size=E)
    return e_cur, w_cur, cache_e, cache_w, cache_norm, tau


@pytest.mark.parametrize("terms", [1, 2, 4, 3, 5, 6, 7])
def test_score_subsets_follow_table5_terms(terms):
    """Each subset scores a matched branch with exactly its terms (Eq. 9, Table 5)."""
    e_cur, w_cur, cache_e, cache_w, cache_norm, tau = _random_selection_inputs(3)
    l1, l2 = 0.7, 0.4
    sel = O.select_branches(e_cur, w_cur, cache_e, cache_w, cache_norm, tau, l1, l2, False, score_terms=terms)
    T, k = e_cur.shape
    checked = 0
    for i in range(T):
        for p in range(k):
            hits = np.nonzero(cache_e[i] == e_cur[i, p])[0]
            if hits.size == 0:
                assert sel["recompute"][i, p] and not sel["matched"][i, p]
                continue
            q = hits[0]
            w = w_cur[i, p]
            parts = {1: w, 2: l1 * abs(w - cache_w[i, q]), 4: l2 * cache_norm[i, q] / cache_norm[i].sum()}
            s = sum(v for bit, v in parts.items() if terms & bit)
            assert sel["score"][i, p] == pytest.approx(s, rel=1e-12, abs=1e-15)
            assert sel["recompute"][i, p] == (np.float32(s) > np.float32(tau[e_cur[i, p]]))
            checked += 1
    assert checked > 20


def test_all_terms_equals_default_score():
    args = _random_selection_inputs(4)
    a = O.select_branches(*args, 1.0, 0.5, False)
    b = O.select_branches(*args, 1.0, 0.5, False, score_terms=7, granularity="branch")
    for key in ("recompute", "slot", "matched"):
        assert np.array_equal(a[key], b[key])


def test_token_granularity_is_the_or_of_branch_decisions():
    """Token-level reuse (Sec. 3): a token's branches share one decision, which
    recomputes all of them when any branch would be recomputed."""
    e_cur, w_cur, cache_e, cache_w, cache_norm, _ = _random_selection_inputs(5)
    args = (e_cur, w_cur, cache_e, cache_w, cache_norm, np.full(6, 1.0))
    br = O.select_branches(*args, 1.0, 0.5, False)
    tk = O.select_branches(*args, 1.0, 0.5, False, granularity="token")
    anyr = br["recompute"].any(axis=1)
    assert np.array_equal(tk["recompute"], np.repeat(anyr[:, None], br["recompute"].shape[1], axis=1))
    assert np.array_equal(tk["slot"], br["slot"]) and np.array_equal(tk["matched"], br["matched"])
    # Both kinds of token occur, so the rule is exercised.
    assert anyr.any() and (~anyr).any()
    # Every branch of a token carries the token's smallest margin.
    assert np.array_equal(tk["margin"], np.repeat(br["margin"].min(axis=1)[:, None], 3, axis=1))


def test_token_granularity_never_reuses_more_than_branch_granularity():
    e_cur, w_cur, cache_e, cache_w, cache_norm, _ = _random_selection_inputs(6)
    for tau0 in (0.2, 0.5, 0.8, 1.2):
        tau = np.full(6, tau0)
        br = O.select_branches(e_cur, w_cur, cache_e, cache_w, cache_norm, tau, 1.0, 0.5, False)
        tk = O.select_branches(e_cur, w_cur, cache_e, cache_w, cache_norm, tau, 1.0, 0.5, False,
                               granularity="token")
        assert tk["recompute"].sum() >= br["recompute"].sum()
        assert np.all(tk["recompute"] | ~br["recompute"])


# --- Token-level reuse reading of Sec. 4.1 ("reuse cached states") ----------

def _textbook_y(x, w, k):
    return textbook_moe(x, w, k) - x.astype(np.float64)


def test_copy_reading_returns_the_last_computed_output_exactly():
    """Under the "copy" reading a token with an empty recompute set returns
    y^{t0}: its MoE output of the last step it computed one, here the full
    step, which is the textbook Eq. 5 value.  The default reading (Eq. 8)
    instead recombines the cached branches with the current weights."""
    w, x0, rng = tiny_layer(40, T=48, D=16, E=5, k=2, F=10, n_shared=1, bias=True)
    x1 = (x0 + 0.3 * rng.standard_normal(x0.shape)).astype(np.float32)
    x2 = (x1 + 0.1 * rng.standard_normal(x0.shape)).astype(np.float32)
    y0 = _textbook_y(x0, w, 2)
    cur = O.Params(top_k=2, tau0=math.inf)
    cpy = O.Params(top_k=2, tau0=math.inf, token_reuse_policy="copy")
    outs_c, infos_c, _ = _run(w, cpy, [x0, x1, x2], n_shared=1)
    outs_d, infos_d, _ = _run(w, cur, [x0, x1, x2], n_shared=1)
    for t in (1, 2):
        assert np.array_equal(infos_c[t]["recompute"], infos_d[t]["recompute"]), "decisions do not depend on it"
    kept1 = ~infos_c[1]["recompute"].any(axis=1)
    kept12 = kept1 & ~infos_c[2]["recompute"].any(axis=1)
    assert kept1.sum() >= 10 and kept12.sum() >= 5 and (~kept1).sum() >= 3
    # Reused for one and for two steps: still the full step's y, bit for bit
    # the oracle's, and equal to the textbook value.
    np.testing.assert_allclose(outs_c[1][kept1] - x1[kept1], y0[kept1], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(outs_c[2][kept12] - x2[kept12], y0[kept12], rtol=1e-12, atol=1e-12)
    # The current-weight reading differs on those tokens (the weights moved).
    assert np.abs((outs_d[1] - outs_c[1])[kept1]).max() > 1e-6
    # Tokens that computed on step 1 agree under both readings.
    np.testing.assert_array_equal(outs_c[1][~kept1], outs_d[1][~kept1])


def test_copy_reading_after_a_recompute_keeps_the_new_output():
    """A token that recomputes at step 1 and is reused at step 2 returns its
    step-1 output, not the full step's: y^{t0} follows the last computation."""
    w, x0, rng = tiny_layer(41, T=64, D=12, E=4, k=2, F=8)
    prm = O.Params(top_k=2, tau0=0.62, token_reuse_policy="copy")
    xs = [x0]
    for _ in range(2):
        xs.append((xs[-1] + 0.2 * rng.standard_normal(x0.shape)).astype(np.float32))
    outs, infos, _ = _run(w, prm, xs)
    comp1 = infos[1]["recompute"].any(axis=1)
    kept2 = ~infos[2]["recompute"].any(axis=1)
    both = comp1 & kept2
    assert both.sum() >= 3
    y1 = outs[1] - xs[1].astype(np.float64)
    np.testing.assert_allclose((outs[2] - xs[2].astype(np.float64))[both], y1[both], rtol=1e-12, atol=1e-15)
    assert np.abs(y1[both] - _textbook_y(xs[0], w, 2)[both]).max() > 1e-9


def test_copy_reading_equals_default_when_nothing_is_reused():
    w, x0, rng = tiny_layer(42, T=32, D=8, E=4, k=2, F=6)
    xs = [x0, (x0 + 0.3 * rng.standard_normal(x0.shape)).astype(np.float32)]
    a, _, _ = _run(w, O.Params(top_k=2, tau0=-math.inf, token_reuse_policy="copy"), xs)
    b, _, _ = _run(w, O.Params(top_k=2, tau0=-math.inf), xs)
    for oa, ob, x in zip(a, b, xs):
        np.testing.assert_array_equal(oa, ob)
        np.testing.assert_allclose(oa, textbook_moe(x, w, 2), rtol=1e-12, atol=1e-12)
