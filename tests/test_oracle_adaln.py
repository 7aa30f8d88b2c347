"""Pins of the oracle's AdaLN DiT-MoE block (Sec. 3 residual form, cached under
Sec. 4.1) and of its sampler step (Eq. 1) against things other than itself:
torch's float64 layer norm, SiLU, GELU, scaled-dot-product attention and
top-k (library routines) assembled into an independent statement of the block;
the closed form of the DDPM posterior mean; identities of the schedule; and
exact identities of the cached block step (zero gates, repeated inputs, a new
gate reaching reused branches).
"""
import math

import numpy as np
import pytest

from oracle import moeca_oracle as O
from paper_2606_15615_gb300.workloads import tiny_adaln, tiny_attn, tiny_layer

torch = pytest.importorskip("torch")
Fn = pytest.importorskip("torch.nn.functional")


def _t(a):
    return torch.from_numpy(np.asarray(a, np.float64))


# --- pieces ------------------------------------------------------------------

def test_layer_norm_matches_torch_and_its_closed_form():
    rng = np.random.default_rng(1)
    v = rng.standard_normal((7, 24)) * 3.0 + 1.5
    got = O.layer_norm(v, 1e-6)
    ref = Fn.layer_norm(_t(v), (24,), eps=1e-6).numpy()
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(got.mean(axis=1), 0.0, atol=1e-12)
    var = v.var(axis=1)
    np.testing.assert_allclose((got ** 2).mean(axis=1), var / (var + 1e-6), rtol=1e-12)
    # a constant row normalises to 0 (only eps in the denominator)
    assert np.array_equal(O.layer_norm(np.full((1, 8), 3.25), 1e-6), np.zeros((1, 8)))


def test_silu_matches_torch():
    z = np.linspace(-30, 30, 301)
    np.testing.assert_allclose(O.silu(z), Fn.silu(_t(z)).numpy(), rtol=1e-13, atol=1e-300)


def test_modulation_blocks_come_in_shift_scale_gate_order():
    """w_ada = the six scaled identities (j + 1) I stacked: block j of the
    output is (j + 1) SiLU(c); with w_ada = 0 the blocks are b_ada's."""
    D, B = 5, 3
    c = np.random.default_rng(2).standard_normal((B, D))
    w = np.concatenate([(j + 1) * np.eye(D) for j in range(6)])
    mod = O.adaln_modulation(c, w)
    for j in range(6):
        np.testing.assert_allclose(mod[:, j], (j + 1) * O.silu(c), rtol=1e-15)
    b = np.arange(6 * D, dtype=np.float64)
    mod = O.adaln_modulation(c, np.zeros((6 * D, D)), b)
    for j in range(6):
        np.testing.assert_array_equal(mod[:, j], np.broadcast_to(b[j * D:(j + 1) * D], (B, D)))


def test_token_rows_follow_samples():
    vec = np.arange(6.0).reshape(3, 2)
    np.testing.assert_array_equal(O.token_rows(vec, 6, 2), [[0, 1], [0, 1], [2, 3], [2, 3], [4, 5], [4, 5]])
    with pytest.raises(ValueError):
        O.token_rows(vec, 5, 2)


# --- the block against an independent statement --------------------------------

def _adaln_block(seed, T=16, S=8, D=16, H=2, E=4, k=2, F=12, n_shared=0, wscale=0.3, **prm_kw):
    w, x0, rng = tiny_layer(seed, T, D, E, k, F, n_shared=n_shared, bias=True)
    w.update(tiny_attn(seed, D))
    w.update(tiny_adaln(seed, D, wscale=wscale))
    prm = O.Params(top_k=k, n_heads=H, seq_len=S, adaln=True, **prm_kw)
    c = rng.standard_normal((T // S, D))
    return w, x0.astype(np.float64), c, rng, prm


def _torch_block(x, c, w, H, S, k, n_shared):
    """The AdaLN DiT-MoE block without any cache, written with torch library
    routines in float64: layer_norm, silu, scaled_dot_product_attention,
    softmax + topk, gelu(tanh) and dense per-expert einsums."""
    X = _t(x)
    T, D = X.shape
    B = T // S
    mod = Fn.silu(_t(c)) @ _t(w["w_ada"]).T + _t(w["b_ada"])
    mod = mod.reshape(B, 6, D).repeat_interleave(S, dim=0)           # [T, 6, D]
    sh_a, sc_a, g_a, sh_m, sc_m, g_m = mod.unbind(1)
    hin = Fn.layer_norm(X, (D,), eps=1e-6) * (1 + sc_a) + sh_a
    qkv = hin @ _t(w["w_qkv"]).T + _t(w["b_qkv"])
    q, kk, v = qkv.split(D, dim=1)
    dh = D // H
    heads = lambda z: z.reshape(B, S, H, dh).transpose(1, 2)         # noqa: E731
    A = Fn.scaled_dot_product_attention(heads(q), heads(kk), heads(v)).transpose(1, 2).reshape(T, D)
    a = A @ _t(w["w_o"]).T + _t(w["b_o"])
    u = X + g_a * a
    m = Fn.layer_norm(u, (D,), eps=1e-6) * (1 + sc_m) + sh_m
    p = torch.softmax(m @ _t(w["w_gate"]).T + _t(w["b_gate"]), dim=1)
    top_p, top_e = torch.topk(p, k, dim=1)
    wt = top_p / top_p.sum(dim=1, keepdim=True)
    hmid = Fn.gelu(torch.einsum("td,efd->tef", m, _t(w["w1"])), approximate="tanh")
    Y = torch.einsum("tef,edf->ted", hmid, _t(w["w2"]))                # every expert on every token
    y = (wt[:, :, None] * Y[torch.arange(T)[:, None], top_e]).sum(dim=1)
    for s in range(n_shared):
        y = y + Fn.gelu(m @ _t(w["ws1"][s]).T, approximate="tanh") @ _t(w["ws2"][s]).T
    return (u + g_m * y).numpy(), a.numpy(), u.numpy(), m.numpy()


@pytest.mark.parametrize("n_shared", [0, 1])
def test_full_step_matches_independent_torch_block(n_shared):
    w, x, c, _, prm = _adaln_block(21 + n_shared, n_shared=n_shared)
    T, D = x.shape
    mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
    st = O.LayerState.empty(T, D, 4, 2, n_shared, attention=True)
    out, st1, info = O.adaln_block_step(st, x, mod, w, prm, refresh=True)
    ref, a, u, m = _torch_block(x, c, w, prm.n_heads, prm.seq_len, 2, n_shared)
    np.testing.assert_allclose(st1.attn_a, a, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(info["u"], u, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(info["m"], m, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)


def test_zero_gates_pass_the_input_through():
    """gate_a = gate_m = 0 (rows 2D..3D and 5D..6D of w_ada and b_ada zero):
    u = x and out = x exactly, on full and cache steps, while the caches fill."""
    w, x, c, rng, prm = _adaln_block(23, attn_policy="sync", tau0=0.7)
    T, D = x.shape
    for j in (2, 5):
        w["w_ada"][j * D:(j + 1) * D] = 0
        w["b_ada"][j * D:(j + 1) * D] = 0
    mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    for step in range(3):
        out, st, info = O.adaln_block_step(st, x, mod, w, prm, refresh=step == 0)
        np.testing.assert_array_equal(out, x)
        np.testing.assert_array_equal(info["u"], x)
        assert np.abs(st.cache_h).sum() > 0
        x = x + 0.1 * rng.standard_normal(x.shape)


def test_repeated_input_all_reuse_reproduces_the_full_step():
    """Same x and c with tau0 = +inf: nothing is recomputed and the output
    repeats the full step's exactly (sync and stale)."""
    for policy in ("sync", "stale"):
        w, x, c, _, prm = _adaln_block(24, attn_policy=policy, tau0=math.inf)
        T, D = x.shape
        mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
        st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
        out0, st1, _ = O.adaln_block_step(st, x, mod, w, prm, refresh=True)
        out1, _, info = O.adaln_block_step(st1, x, mod, w, prm, refresh=False)
        assert not info["recompute"].any() and len(info["attn_rows"]) == 0
        np.testing.assert_array_equal(out1, out0)


def test_new_gates_reach_reused_branches():
    """Only gate_m changes between the steps and every branch is reused: the
    output moves by (g_new - g_old) * y with y the cached combine, so the
    caches hold ungated outputs and the current gate applies."""
    w, x, c, _, prm = _adaln_block(25, attn_policy="sync", tau0=math.inf)
    T, D = x.shape
    mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    out0, st1, info0 = O.adaln_block_step(st, x, mod, w, prm, refresh=True)
    mod2 = mod.copy()
    mod2[:, 5] = mod[:, 5] * -1.5 + 0.25
    out1, _, info1 = O.adaln_block_step(st1, x, mod2, w, prm, refresh=False)
    assert not info1["recompute"].any()
    g0 = O.token_rows(mod[:, 5], T, prm.seq_len)
    g1 = O.token_rows(mod2[:, 5], T, prm.seq_len)
    y = (out0 - info0["u"]) / g0
    np.testing.assert_allclose(out1, info1["u"] + g1 * y, rtol=1e-12, atol=1e-12)


def test_all_recompute_cache_step_equals_full_step_inputs():
    """tau0 = -inf: every token recomputes its attention, so a, u and the FFN
    input m equal the full step's on the new x (the routing differs: the
    cache step routes on m' from a^{t0})."""
    w, x, c, rng, prm = _adaln_block(26, attn_policy="sync", tau0=-math.inf)
    T, D = x.shape
    mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    _, st1, _ = O.adaln_block_step(st, x, mod, w, prm, refresh=True)
    x1 = x + 0.2 * rng.standard_normal(x.shape)
    _, st2, info = O.adaln_block_step(st1, x1, mod, w, prm, refresh=False)
    _, st3, ref = O.adaln_block_step(st1, x1, mod, w, prm, refresh=True)
    assert len(info["attn_rows"]) == T
    np.testing.assert_array_equal(st2.attn_a, st3.attn_a)
    np.testing.assert_array_equal(info["u"], ref["u"])
    np.testing.assert_array_equal(info["m"], ref["m"])
    g_a = O.token_rows(mod[:, 2], T, prm.seq_len)
    np.testing.assert_array_equal(info["route_in"],
                                  O.modulate(O.layer_norm(x1 + g_a * st1.attn_a, 1e-6),
                                             O.token_rows(mod[:, 3], T, prm.seq_len),
                                             O.token_rows(mod[:, 4], T, prm.seq_len)))


def test_sync_rule_mixes_kept_and_recomputed_tokens_in_bf16():
    w, x, c, rng, prm = _adaln_block(27, attn_policy="sync", tau0=0.62, act_store="bf16")
    T, D = x.shape
    x = O.round_bf16(x)
    mod = O.adaln_modulation(c, w["w_ada"], w["b_ada"])
    st = O.LayerState.empty(T, D, 4, 2, 0, attention=True)
    _, st1, _ = O.adaln_block_step(st, x, mod, w, prm, refresh=True)
    x1 = O.round_bf16(x + 0.3 * rng.standard_normal(x.shape))
    _, st2, info = O.adaln_block_step(st1, x1, mod, w, prm, refresh=False)
    act = info["token_any"]
    assert 0 < act.sum() < T
    np.testing.assert_array_equal(st2.attn_a[~act], st1.attn_a[~act])
    np.testing.assert_array_equal(info["m"][~act], info["route_in"][~act])
    assert (info["m"][act] != info["route_in"][act]).any()
    for v in (info["h"], info["u"], info["m"], st2.attn_a):
        np.testing.assert_array_equal(v, O.round_bf16(v))


def test_stack_applies_each_layers_modulation():
    w, x, c, rng, prm = _adaln_block(28, attn_policy="sync", tau0=0.62, refresh_period=2)
    w2 = dict(w)
    w2.update(tiny_adaln(99, x.shape[1], wscale=0.3))
    stack = O.Stack([w, w2], prm, hidden=x.shape[1], n_experts=4)
    out, infos = stack.step(x, 0, cond=c)
    assert not np.array_equal(infos[0]["mod"], infos[1]["mod"])
    np.testing.assert_array_equal(infos[1]["mod"], O.adaln_modulation(c, w2["w_ada"], w2["b_ada"]))


# --- sampler (Eq. 1) -------------------------------------------------------------

def test_schedule_identities():
    t, alpha, abar, beta = O.ddpm_schedule(1000)
    betas = np.linspace(1e-4, 0.02, 1000)
    np.testing.assert_array_equal(t, np.arange(1000))
    np.testing.assert_allclose(beta, betas, rtol=1e-9, atol=1e-15)     # unrespaced: the training betas
    t, alpha, abar, beta = O.ddpm_schedule(250)
    assert t[0] == 0 and t[-1] == 999 and np.all(np.diff(t) > 0)
    np.testing.assert_allclose(np.cumprod(alpha), abar, rtol=1e-12)    # the respaced alphas rebuild abar
    np.testing.assert_allclose(abar[-1], np.prod(1 - betas), rtol=1e-12)
    assert np.all((beta > 0) & (beta < 1))


def test_reverse_mean_equals_the_posterior_mean_given_the_true_noise():
    """With eps the noise that made x_t from x_0 (x_t = sqrt(abar_t) x_0 +
    sqrt(1 - abar_t) eps), Eq. 1's mean equals the Gaussian posterior mean
    of x_{t-1} given (x_t, x_0):
      sqrt(abar_{t-1}) beta_t / (1 - abar_t) x_0
      + sqrt(alpha_t) (1 - abar_{t-1}) / (1 - abar_t) x_t."""
    _, alpha, abar, beta = O.ddpm_schedule(50)
    rng = np.random.default_rng(4)
    x0 = rng.standard_normal(64)
    eps = rng.standard_normal(64)
    for j in range(1, 50):
        xt = math.sqrt(abar[j]) * x0 + math.sqrt(1 - abar[j]) * eps
        got = O.ddpm_step(xt, eps, np.zeros(64), alpha[j], abar[j], 0.0)
        post = (math.sqrt(abar[j - 1]) * beta[j] / (1 - abar[j]) * x0
                + math.sqrt(alpha[j]) * (1 - abar[j - 1]) / (1 - abar[j]) * xt)
        np.testing.assert_allclose(got, post, rtol=1e-10, atol=1e-12)


def test_noise_term_scales_with_sigma():
    got = O.ddpm_step(np.zeros(4), np.zeros(4), np.array([1.0, -2.0, 0.5, 0.0]), 0.9, 0.5, math.sqrt(0.1))
    np.testing.assert_allclose(got, math.sqrt(0.1) * np.array([1.0, -2.0, 0.5, 0.0]), rtol=1e-15)


# --- planted mistakes: each must fail a pin above ----------------------------------

def _mut_modulate_swapped(v, shift, scale):
    return np.asarray(v, np.float64) * (1.0 + np.asarray(shift, np.float64)) + np.asarray(scale, np.float64)


def _mut_ln_unbiased(v, eps):
    v = np.asarray(v, np.float64)
    mu = v.mean(axis=-1, keepdims=True)
    var = ((v - mu) ** 2).sum(axis=-1, keepdims=True) / (v.shape[-1] - 1)
    return (v - mu) / np.sqrt(var + eps)


def _mut_ddpm_no_sqrt(x_t, eps, z, alpha_t, alpha_bar_t, sigma_t):
    x_t = np.asarray(x_t, np.float64)
    return (x_t - (1.0 - alpha_t) / (1.0 - alpha_bar_t) * np.asarray(eps, np.float64)) / math.sqrt(alpha_t) \
        + sigma_t * np.asarray(z, np.float64)


_REAL_RC = O.recompute_and_combine


def _mut_gate_ignored(*args, resid=None, gate=None, **kw):
    return _REAL_RC(*args, resid=resid, gate=None, **kw)


_REAL_ATTN = O.attention


def _mut_attention_on_raw_input(h, *args, **kw):
    # An attention sub-layer that reads something other than the normalised,
    # modulated h: here h rescaled and shifted, as the raw block input would be.
    return _REAL_ATTN(np.asarray(h) * 3.0 + 1.0, *args, **kw)


PLANTED = {
    "shift_scale_swapped": ("modulate", _mut_modulate_swapped),
    "unbiased_variance": ("layer_norm", _mut_ln_unbiased),
    "gate_not_applied": ("recompute_and_combine", _mut_gate_ignored),
    "attention_input_not_normalised": ("attention", _mut_attention_on_raw_input),
    "eps_coefficient_without_sqrt": ("ddpm_step", _mut_ddpm_no_sqrt),
}


@pytest.mark.parametrize("name", list(PLANTED))
def test_planted_mistake_fails_a_pin(name, monkeypatch):
    attr, fn = PLANTED[name]
    monkeypatch.setattr(O, attr, fn)
    pins = [lambda: test_layer_norm_matches_torch_and_its_closed_form(),
            lambda: test_full_step_matches_independent_torch_block(0),
            lambda: test_new_gates_reach_reused_branches(),
            lambda: test_reverse_mean_equals_the_posterior_mean_given_the_true_noise(),
            lambda: test_golden_values()]
    failed = 0
    for pin in pins:
        try:
            pin()
        except AssertionError:
            failed += 1
    assert failed >= 1, f"planted mistake {name} passed every pin"


def test_golden_values():
    """The hand-worked fixture (tests/golden/adaln_ddpm.json) through this module's view of the oracle."""
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "adaln_ddpm.json")) as f:
        g = json.load(f)
    d = g["ddpm"]
    np.testing.assert_allclose(O.ddpm_step(d["x_t"], d["eps"], d["z"], d["alpha"], d["alpha_bar"], d["sigma"]),
                               d["x_prev"], rtol=1e-14)
    m = g["layer_norm_modulate"]
    got = O.modulate(O.layer_norm(np.array([m["v"]]), m["eps"]), np.array(m["shift"]), np.array(m["scale"]))
    np.testing.assert_allclose(got[0], m["out"], rtol=1e-14, atol=1e-15)
