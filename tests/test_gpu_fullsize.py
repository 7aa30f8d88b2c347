"""Full-size workloads, in the launch configuration bench.py times (marked gpu).

For each bf16 workload at its full shape (T, D, E, k, F, L), a few trajectory
steps run through the C ABI with on-device seeded weights.  On a cache step,
three layers (first, middle, last) are checked against the oracle:
  * EMA statistic, thresholds and every group's row list: over all tokens;
  * routing, recompute decisions, slots and the layer output: on a sample of
    tokens the oracle computes one by one (teacher-forced, see gpu_harness).
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_harness import NEAR, check_gate_weights, expected_lists, np_of, params_of, rel_l2  # noqa: E402
from oracle import moeca_oracle as O  # noqa: E402
from paper_2606_15615_gb300 import workloads as W  # noqa: E402


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA GPU is required for gpu-marked tests")
    from paper_2606_15615_gb300 import build
    build.build()
    from paper_2606_15615_gb300 import moeca
    return moeca


def _take(st, rows):
    idx = torch.as_tensor(rows, device="cuda", dtype=torch.long)
    return {k: (None if v is None or k == "n_tokens" else np_of(v.index_select(0, idx)).astype(np.float64))
            for k, v in st.items()}


@pytest.mark.parametrize("index", [2, 3, 4, 5])
def test_fullsize_sampled_parity(M, index):
    wl = W.workload(index)
    dev = torch.device("cuda", 0)
    weights = [W.make_layer_weights_device(wl, l, dev) for l in range(wl.n_layers)]
    cfg = M.moeca_config_default(n_layers=wl.n_layers, hidden=wl.hidden, ffn=wl.ffn, n_experts=wl.n_experts,
                                 top_k=wl.top_k, n_shared=wl.n_shared, max_tokens=wl.n_tokens,
                                 dtype=M.MOECA_BF16, refresh_period=wl.refresh_period,
                                 tau0=0.75 if wl.top_k == 2 else 0.2)
    stack = M.Stack(cfg, weights)
    T, k, E, S = wl.n_tokens, wl.top_k, wl.n_experts, wl.n_shared
    xs = [torch.from_numpy(x).to(dev).to(torch.bfloat16) for x in W.trajectory(wl, 3)]
    stack.step(xs[0], 0)
    stack.step(xs[1], 1)
    layers = sorted({0, wl.n_layers // 2, wl.n_layers - 1})
    pre = {l: stack.get_state(l) for l in layers}
    pre = {l: {kk: (v.clone() if isinstance(v, torch.Tensor) else v) for kk, v in s.items()} for l, s in pre.items()}
    out = stack.step(xs[2], 2)
    torch.cuda.synchronize()
    prm = params_of(cfg)
    rng = np.random.default_rng(index)
    sample = np.sort(rng.choice(T, size=48, replace=False))
    for l in layers:
        tr = stack.get_trace(l, T)
        post = stack.get_state(l)
        w = {kk: (None if v is None else np_of(v)) for kk, v in weights[l].items()}
        # EMA and thresholds over all tokens.
        e_g = np_of(tr["route_e"]).astype(np.int64)
        C_o = O.ema_update(np_of(pre[l]["ema"]).astype(np.float64).T, e_g, prm.beta)
        C_g = np_of(post["ema"]).astype(np.float64).T
        assert np.allclose(C_g, C_o, rtol=2e-6, atol=1e-7)
        tau_o = O.expert_threshold(O.normalized_entropy(C_g), prm.tau0, prm.alpha)
        tau_g = np_of(tr["tau"]).astype(np.float64)
        assert np.allclose(tau_g, tau_o, rtol=1e-5, atol=1e-6)
        # Row lists over all tokens, from the GPU decisions.
        rec_all = np_of(tr["recompute"]).astype(bool)
        slot_all = np_of(tr["slot"]).astype(np.int64)
        any_all = np_of(tr["token_any"]).astype(bool)
        cnt, off, flat = expected_lists(e_g, rec_all, slot_all, any_all, E, k, S, False, False)
        assert np.array_equal(np_of(tr["counts"]), cnt) and np.array_equal(np_of(tr["offsets"]), off)
        assert np.array_equal(np_of(tr["list"])[: off[-1]], flat)
        assert 0 < rec_all.sum() < rec_all.size, "a cache step with both kinds of branch"
        # Sampled tokens: routing, decisions, output.
        u = np_of(tr["layer_in"])[sample].astype(np.float64)
        e_o, w_o, near, cond = O.route(u, w["w_gate"], w.get("b_gate"), k, prm.renorm_topk)
        ok = near >= NEAR
        assert np.array_equal(e_o[ok], e_g[sample][ok])
        w_g = np_of(tr["route_w"]).astype(np.float64)[sample]
        check_gate_weights(w_g[ok], w_o[ok], cond[ok])
        ps = _take(pre[l], sample)
        sel = O.select_branches(e_g[sample], w_g, ps["cache_e"].astype(np.int64), ps["cache_w"], ps["cache_norm"],
                                tau_g, prm.lambda1, prm.lambda2, False)
        far = sel["margin"] >= NEAR
        assert np.array_equal(sel["slot"], slot_all[sample])
        assert not (far & (sel["recompute"] != rec_all[sample])).any()
        st_o = O.LayerState(ps["cache_e"].astype(np.int32), ps["cache_w"], ps["cache_norm"], ps["cache_h"],
                            ps["shared_h"], np.zeros((E, len(sample))), True)
        wo = dict(w)
        wo["ws1"] = None if w["ws1"] is None else w["ws1"]
        out_o, new_o, _ = O.recompute_and_combine(st_o, u, e_g[sample], w_g, rec_all[sample], slot_all[sample],
                                                  wo, prm, False)
        if l + 1 < wl.n_layers:
            got = np_of(stack.get_trace(l + 1, T)["layer_in"])[sample]
        else:
            got = np_of(out)[sample]
        assert rel_l2(got, out_o) <= 1e-2
        # Without a norm between layers the residual stream grows with depth, so
        # the absolute bound applies to outputs normalised by their RMS.
        scale = max(1.0, float(np.sqrt(np.mean(out_o ** 2))))
        assert float(np.abs(got - out_o).max()) <= 5e-2 * scale
    stack.close()
