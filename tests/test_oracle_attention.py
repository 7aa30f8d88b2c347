"""Pins of the oracle's attention path (Sec. 4.1: cached attention output a_i
and the synchronized MoE / attention update) against things other than itself:
torch's fp64 scaled-dot-product attention (a library routine), closed forms of
degenerate cases, invariants of self-attention, torch's bf16 conversion, and
identities of the block step (zero attention reduces to the MoE layer; a
repeated input reproduces the full step or the previous output exactly).
"""
import math

import numpy as np
import pytest

from oracle import moeca_oracle as O
from paper_2606_15615_gb300.workloads import tiny_attn, tiny_layer

torch = pytest.importorskip("torch")


def _sdpa_ref(x, aw, H, S):
    """Multi-head attention through torch.nn.functional.scaled_dot_product_attention
    in float64, sample by sample (an implementation independent of the oracle)."""
    import torch.nn.functional as Fn
    X = torch.from_numpy(np.asarray(x, np.float64))
    T, D = X.shape
    dh = D // H
    Wqkv = torch.from_numpy(aw["w_qkv"].astype(np.float64))
    qkv = X @ Wqkv.T
    if aw["b_qkv"] is not None:
        qkv = qkv + torch.from_numpy(aw["b_qkv"].astype(np.float64))
    q, k, v = qkv.split(D, dim=1)
    outs = []
    for b in range(T // S):
        sl = slice(b * S, (b + 1) * S)
        heads = lambda t: t[sl].reshape(S, H, dh).transpose(0, 1)  # noqa: E731
        o = Fn.scaled_dot_product_attention(heads(q)[None], heads(k)[None], heads(v)[None])[0]
        outs.append(o.transpose(0, 1).reshape(S, D))
    A = torch.cat(outs)
    a = A @ torch.from_numpy(aw["w_o"].astype(np.float64)).T
    if aw["b_o"] is not None:
        a = a + torch.from_numpy(aw["b_o"].astype(np.float64))
    return a.numpy()


@pytest.mark.parametrize("T,S,D,H,bias", [(24, 8, 16, 2, True), (12, 12, 24, 3, False), (18, 6, 36, 4, True)])
def test_attention_matches_torch_sdpa(T, S, D, H, bias):
    aw = tiny_attn(T + D, D, bias=bias, wscale=0.4)
    x = np.random.default_rng(T * D).standard_normal((T, D))
    got = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S)
    np.testing.assert_allclose(got, _sdpa_ref(x, aw, H, S), rtol=1e-12, atol=1e-12)


def test_attention_row_subset_equals_rows_of_full():
    D, H, S, T = 16, 4, 5, 20
    aw = tiny_attn(3, D)
    x = np.random.default_rng(3).standard_normal((T, D))
    full = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S)
    rows = np.array([0, 4, 5, 11, 19])
    sub = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S, rows)
    np.testing.assert_allclose(sub, full[rows], rtol=0, atol=1e-14)


def test_one_token_samples_reduce_to_value_and_output_projections():
    """seq_len = 1: the softmax over a single key is 1, so a = (x Wv^T + bv) Wo^T + bo."""
    D, H, T = 12, 3, 7
    aw = tiny_attn(4, D)
    x = np.random.default_rng(4).standard_normal((T, D))
    got = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, 1)
    wv = aw["w_qkv"][2 * D:].astype(np.float64)
    v = x @ wv.T + aw["b_qkv"][2 * D:]
    np.testing.assert_allclose(got, v @ aw["w_o"].astype(np.float64).T + aw["b_o"], rtol=1e-12, atol=1e-13)


def test_zero_queries_give_the_sample_mean_of_the_values():
    """Wq = 0 and bq = 0: every score is 0, the softmax is uniform over the
    sample's keys, and every token of a sample gets mean(V) Wo^T + bo."""
    D, H, S, T = 8, 2, 4, 12
    aw = tiny_attn(5, D)
    aw["w_qkv"][:D] = 0.0
    aw["b_qkv"][:D] = 0.0
    x = np.random.default_rng(5).standard_normal((T, D))
    got = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S)
    v = x @ aw["w_qkv"][2 * D:].astype(np.float64).T + aw["b_qkv"][2 * D:]
    for b in range(T // S):
        mean = v[b * S:(b + 1) * S].mean(axis=0) @ aw["w_o"].astype(np.float64).T + aw["b_o"]
        np.testing.assert_allclose(got[b * S:(b + 1) * S], np.broadcast_to(mean, (S, D)), rtol=1e-12, atol=1e-13)


def test_permutation_within_a_sample_permutes_outputs_and_samples_are_isolated():
    D, H, S, T = 16, 2, 6, 18
    aw = tiny_attn(6, D)
    rng = np.random.default_rng(6)
    x = rng.standard_normal((T, D))
    a = O.attention(x, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S)
    perm = np.arange(T)
    perm[S:2 * S] = S + rng.permutation(S)
    x2 = x[perm].copy()
    x2[2 * S:] = rng.standard_normal((S, D))          # another sample changes
    a2 = O.attention(x2, aw["w_qkv"], aw["b_qkv"], aw["w_o"], aw["b_o"], H, S)
    np.testing.assert_allclose(a2[:2 * S], a[perm][:2 * S], rtol=1e-12, atol=1e-13)
    assert np.abs(a2[2 * S:] - a[2 * S:]).max() > 1e-3


def test_round_bf16_matches_torch_conversion():
    rng = np.random.default_rng(7)
    vals = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.integers(-6, 6, 4000),
                           [1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -9, -(1.0 + 2.0 ** -8), 0.0, -0.0,
                            np.inf, -np.inf, 3.0e38]])
    ref = torch.from_numpy(vals.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    got = O.round_bf16(vals)
    assert np.array_equal(got, ref)
    assert got[4000] == 1.0 and got[4001] == 1.0 + 2.0 ** -7   # ties to even; above the tie rounds up


# --- block step (attention sub-layer, then MoE sub-layer) ---------------------

def _block(seed, T=16, S=8, D=16, H=2, E=4, k=2, F=12, n_shared=0, **prm_kw):
    w, x0, rng = tiny_layer(seed, T, D, E, k, F, n_shared=n_shared, bias=True)
    w.update(tiny_attn(seed, D))
    prm = O.Params(top_k=k, n_heads=H, seq_len=S, **prm_kw)
    return w, x0, rng, prm


def test_zero_attention_block_is_the_moe_layer():
    """Wo = 0 and bo = 0 make a = 0, so every policy's block step is the MoE
    layer step on x, on full and cache steps alike."""
    for policy in ("sync", "stale", "full"):
        w, x0, rng, prm = _block(11, attn_policy=policy, tau0=0.7)
        w["w_o"] = np.zeros_like(w["w_o"])
        w["b_o"] = np.zeros_like(w["b_o"])
        T, D = x0.shape
        sb = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
        sm = O.LayerState.empty(T, D, 4, 2, 0)
        x = x0.astype(np.float64)
        for step in range(3):
            ob, sb, ib = O.block_step(sb, x, w, prm, refresh=(step == 0))
            om, sm, im = O.layer_step(sm, x, w, prm, refresh=(step == 0))
            assert np.array_equal(ob, om)
            assert np.array_equal(ib["recompute"], im["recompute"])
            x = x + 0.05 * rng.standard_normal(x.shape)


def test_repeated_input_all_recompute_equals_full_step():
    """Same x at a cache step with tau0 = -inf: every branch and every token's
    attention is recomputed, and u' = x + a^{t0} equals the fresh u, so the
    sync step reproduces the full step bit for bit."""
    w, x0, _, prm = _block(12, attn_policy="sync", tau0=-math.inf)
    T, D = x0.shape
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    out0, st1, _ = O.block_step(st, x0, w, prm, refresh=True)
    out1, st2, info = O.block_step(st1, x0, w, prm, refresh=False)
    assert info["recompute"].all() and len(info["attn_rows"]) == T
    ref, _, _ = O.block_step(st1, x0, w, prm, refresh=True)
    np.testing.assert_array_equal(out1, ref)
    np.testing.assert_array_equal(st2.attn_a, st1.attn_a)


def test_repeated_input_all_reuse_returns_previous_output():
    """Same x with tau0 = +inf: every branch matches and is reused, no token
    recomputes attention, and the output repeats the previous one exactly."""
    for policy in ("sync", "stale"):
        w, x0, _, prm = _block(13, attn_policy=policy, tau0=math.inf)
        T, D = x0.shape
        st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
        out0, st1, _ = O.block_step(st, x0, w, prm, refresh=True)
        out1, st2, info = O.block_step(st1, x0, w, prm, refresh=False)
        assert not info["recompute"].any() and len(info["attn_rows"]) == 0
        np.testing.assert_array_equal(out1, out0)


def test_sync_updates_attention_exactly_on_tokens_with_recomputed_branches():
    w, x0, rng, prm = _block(14, attn_policy="sync", tau0=0.62, act_store="bf16")
    T, D = x0.shape
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    _, st, _ = O.block_step(st, x0, w, prm, refresh=True)
    x1 = O.round_bf16(x0 + 0.3 * rng.standard_normal(x0.shape))
    _, st2, info = O.block_step(st, x1, w, prm, refresh=False)
    act = info["token_any"]
    assert 0 < act.sum() < T, "the case should mix tokens with and without recomputed branches"
    np.testing.assert_array_equal(st2.attn_a[~act], st.attn_a[~act])
    fresh = O.round_bf16(O.attention(x1, w["w_qkv"], w["b_qkv"], w["w_o"], w["b_o"], 2, 8))
    np.testing.assert_array_equal(st2.attn_a[act], fresh[act])
    # router input keeps the cached attention; the MoE input takes the fresh rows
    np.testing.assert_array_equal(info["route_in"], O.round_bf16(x1 + st.attn_a))
    np.testing.assert_array_equal(info["u"][act], O.round_bf16(x1[act] + fresh[act]))
    np.testing.assert_array_equal(info["u"][~act], info["route_in"][~act])


def test_stale_policy_keeps_attention_from_the_full_step():
    w, x0, rng, prm = _block(15, attn_policy="stale", tau0=0.62)
    T, D = x0.shape
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    _, st, _ = O.block_step(st, x0, w, prm, refresh=True)
    a0 = st.attn_a.copy()
    x = x0.astype(np.float64)
    for _ in range(3):
        x = x + 0.3 * rng.standard_normal(x.shape)
        _, st, info = O.block_step(st, x, w, prm, refresh=False)
        np.testing.assert_array_equal(st.attn_a, a0)
        np.testing.assert_array_equal(info["u"], x + a0)


def test_full_policy_cache_step_routes_on_fresh_attention():
    w, x0, rng, prm = _block(16, attn_policy="full", tau0=0.62)
    T, D = x0.shape
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    _, st, _ = O.block_step(st, x0, w, prm, refresh=True)
    x1 = x0 + 0.3 * rng.standard_normal(x0.shape)
    out, st2, info = O.block_step(st, x1, w, prm, refresh=False)
    a = O.attention(x1, w["w_qkv"], w["b_qkv"], w["w_o"], w["b_o"], 2, 8)
    np.testing.assert_allclose(st2.attn_a, a, rtol=0, atol=0)
    np.testing.assert_array_equal(info["route_in"], x1 + a)
    ref_out, _, ref_info = O.layer_step(st, x1 + a, w, prm, refresh=False)
    np.testing.assert_array_equal(out, ref_out)


def test_stack_with_heads_runs_blocks():
    w, x0, rng, prm = _block(17, attn_policy="sync", tau0=0.62, refresh_period=3)
    T, D = x0.shape
    stack = O.Stack([w, w], prm, hidden=D, n_experts=4)
    x = x0
    for t in range(4):
        out, infos = stack.step(x, t)
        assert all("attn_rows" in i for i in infos)
        assert (len(infos[0]["attn_rows"]) == T) == (t % 3 == 0)
        x = x + 0.1 * rng.standard_normal(x.shape)
