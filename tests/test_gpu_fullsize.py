"""Full-size workloads, in the launch configuration bench.py times (marked gpu).

For each bf16 workload at its full shape (T, D, E, k, F, L), tau0 is
calibrated on the GPU to the reuse points the benchmark reports (0/30/60/90%
for the 12-layer D 768 stack, 0/30/60/95% for the 64-expert layer, 60% for
the others), then four trajectory steps run through the C ABI with on-device
seeded weights.  On the last (cache) step three layers (first, middle, last)
are checked against the oracle:
  * EMA statistic, thresholds and every group's row list: over all tokens;
  * routing, recompute decisions, slots and the layer output: on 256 sampled
    tokens the oracle computes one by one (teacher-forced, see gpu_harness),
    with the near-margin exclusions counted and bounded and the outputs held
    to the relative L2 and per-element max-abs bounds of the harness.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_harness import (NEAR, REPORTS, Report, assert_margins, check_gate_weights, check_output,  # noqa: E402
                         count_route_margins, expected_lists, fresh_terms, np_of, params_of)
from oracle import moeca_oracle as O  # noqa: E402
from paper_2606_15615_gb300 import workloads as W  # noqa: E402

N_SAMPLE = 256
POINTS = {2: [0.0, 0.3, 0.6, 0.9], 3: [0.6], 4: [0.6], 5: [0.0, 0.3, 0.6, 0.95]}
CASES = [(i, r) for i in (2, 3, 4, 5) for r in POINTS[i]]


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA GPU is required for gpu-marked tests")
    from paper_2606_15615_gb300 import build
    build.build()
    from paper_2606_15615_gb300 import moeca
    return moeca


_STACKS = {}


def _stack(M, index):
    """One handle per workload for the module (the weights are large)."""
    if index not in _STACKS:
        for old in list(_STACKS):
            _STACKS.pop(old)[0].close()
        wl = W.workload(index)
        dev = torch.device("cuda", 0)
        weights = [W.make_layer_weights_device(wl, l, dev) for l in range(wl.n_layers)]
        cfg = M.moeca_config_default(n_layers=wl.n_layers, hidden=wl.hidden, ffn=wl.ffn, n_experts=wl.n_experts,
                                     top_k=wl.top_k, n_shared=wl.n_shared, max_tokens=wl.n_tokens,
                                     dtype=M.MOECA_BF16, refresh_period=wl.refresh_period)
        xs = [torch.from_numpy(x).to(dev).to(torch.bfloat16) for x in W.trajectory(wl, 4)]
        _STACKS[index] = (M.Stack(cfg, weights), cfg, weights, xs, wl)
    return _STACKS[index]


def _run(M, st, xs, tau0, upto):
    M.moeca_reset(st.handle)
    for t in range(upto):
        st.step(xs[t], t, tau0=tau0)
        if t == 0:
            torch.cuda.synchronize()
            M.moeca_reset_stats(st.handle)


def _calibrate(M, st, xs, target):
    """tau0 whose reuse over cache steps 1..3 is closest to ``target`` (bisection)."""
    if target <= 0.0:
        return -math.inf

    def reuse(tau0):
        _run(M, st, xs, tau0, 4)
        s = st.stats()
        return s["reused"] / max(s["branches"], 1)

    lo, hi = 0.0, 4.0
    best = (hi, reuse(hi))
    if best[1] <= target:
        return hi
    for _ in range(12):
        mid = 0.5 * (lo + hi)
        r = reuse(mid)
        if abs(r - target) < abs(best[1] - target):
            best = (mid, r)
        lo, hi = (mid, hi) if r < target else (lo, mid)
    return best[0]


def _take(st, rows):
    idx = torch.as_tensor(rows, device="cuda", dtype=torch.long)
    return {k: (None if v is None or k == "n_tokens" else np_of(v.index_select(0, idx)).astype(np.float64))
            for k, v in st.items()}


@pytest.mark.parametrize("index,target", CASES, ids=[f"cfg{i}-reuse{int(100 * r)}" for i, r in CASES])
def test_fullsize_sampled_parity(M, index, target):
    st, cfg, weights, xs, wl = _stack(M, index)
    T, k, E, S = wl.n_tokens, wl.top_k, wl.n_experts, wl.n_shared
    tau0 = _calibrate(M, st, xs, target)
    _run(M, st, xs, tau0, 3)
    layers = sorted({0, wl.n_layers // 2, wl.n_layers - 1})
    pre = {l: st.get_state(l) for l in layers}
    pre = {l: {kk: (v.clone() if isinstance(v, torch.Tensor) else v) for kk, v in s.items()} for l, s in pre.items()}
    out = st.step(xs[3], 3, tau0=tau0)
    torch.cuda.synchronize()
    s3 = st.stats()
    achieved = s3["reused"] / max(s3["branches"], 1)
    prm = params_of(cfg)
    prm.tau0 = tau0
    rng = np.random.default_rng(100 * index + int(100 * target))
    sample = np.sort(rng.choice(T, size=N_SAMPLE, replace=False))
    rep = Report()
    for l in layers:
        tr = st.get_trace(l, T)
        post = st.get_state(l)
        w = {kk: (None if v is None else np_of(v)) for kk, v in weights[l].items()}
        wo = {kk: (None if v is None else np.asarray(v, np.float64)) for kk, v in w.items()}
        # EMA and thresholds over all tokens.
        e_g = np_of(tr["route_e"]).astype(np.int64)
        C_o = O.ema_update(np_of(pre[l]["ema"]).astype(np.float64).T, e_g, prm.beta)
        C_g = np_of(post["ema"]).astype(np.float64).T
        assert np.allclose(C_g, C_o, rtol=2e-6, atol=1e-7)
        tau_o = O.expert_threshold(O.normalized_entropy(C_g), prm.tau0, prm.alpha)
        tau_g = np_of(tr["tau"]).astype(np.float64)
        if math.isfinite(tau0):
            assert np.allclose(tau_g, tau_o, rtol=1e-5, atol=1e-6)
        else:
            assert np.array_equal(tau_g, tau_o)
        # Row lists over all tokens, from the GPU decisions.
        rec_all = np_of(tr["recompute"]).astype(bool)
        slot_all = np_of(tr["slot"]).astype(np.int64)
        any_all = np_of(tr["token_any"]).astype(bool)
        cnt, off, flat = expected_lists(e_g, rec_all, slot_all, any_all, E, k, S, False, False)
        assert np.array_equal(np_of(tr["counts"]), cnt) and np.array_equal(np_of(tr["offsets"]), off)
        assert np.array_equal(np_of(tr["list"])[: off[-1]], flat)
        if target > 0.0:
            assert 0 < rec_all.sum() < rec_all.size, "a cache step with both kinds of branch"
        else:
            assert rec_all.all()
        # Sampled tokens: routing, decisions, output.
        u = np_of(tr["layer_in"])[sample].astype(np.float64)
        e_o, w_o, ok, cond = count_route_margins(rep, u, wo, k, prm.renorm_topk, e_g[sample])
        assert np.array_equal(e_o[ok], e_g[sample][ok])
        w_g = np_of(tr["route_w"]).astype(np.float64)[sample]
        check_gate_weights(w_g[ok], w_o[ok], cond[ok])
        ps = _take(pre[l], sample)
        sel = O.select_branches(e_g[sample], w_g, ps["cache_e"].astype(np.int64), ps["cache_w"], ps["cache_norm"],
                                tau_g, prm.lambda1, prm.lambda2, False)
        far = sel["margin"] >= NEAR
        rep.near_score += int((~far).sum())
        rep.near_score_diff += int((~far & (sel["recompute"] != rec_all[sample])).sum())
        assert np.array_equal(sel["slot"], slot_all[sample])
        assert np.array_equal(sel["matched"], np_of(tr["matched"]).astype(bool)[sample])
        assert not (far & (sel["recompute"] != rec_all[sample])).any()
        st_o = O.LayerState(ps["cache_e"].astype(np.int32), ps["cache_w"], ps["cache_norm"], ps["cache_h"],
                            ps["shared_h"], np.zeros((E, len(sample))), True)
        rec_s, slot_s = rec_all[sample], slot_all[sample]
        out_o, new_o, _ = O.recompute_and_combine(st_o, u, e_g[sample], w_g, rec_s, slot_s, wo, prm, False)
        if l + 1 < wl.n_layers:
            got = np_of(st.get_trace(l + 1, T)["layer_in"])[sample]
        else:
            got = np_of(out)[sample]
        terms = fresh_terms(u, wo, e_g[sample], w_g, rec_s, slot_s, new_o, prm.gelu, None,
                            rec_s.any(axis=1) if S else None)
        check_output(rep, got, out_o, True, 1e-2, what=f"layer {l} output", terms=terms)
        rep.layers_checked += 1
        rep.branches += N_SAMPLE * k
        rep.recomputed += int(rec_s.sum())
        rep.reused += int((~rec_s).sum())
    rep.steps = 1
    REPORTS.append((f"fullsize cfg{index} reuse {achieved:.2f} (target {target})", rep))
    assert_margins(rep)
    if target == CASES[-1][1] and index == CASES[-1][0]:
        for key in list(_STACKS):
            _STACKS.pop(key)[0].close()
