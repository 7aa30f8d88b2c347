"""GPU vs oracle parity of the AdaLN DiT-MoE block (Sec. 3 residual form
x + AdaLN o f(x), cached under Sec. 4.1) and of the sampler step (Eq. 1),
through the C ABI (marked gpu).

Every layer of every step is teacher-forced (see gpu_harness): the step's
modulation vectors against the oracle's, the attention of h = LN-modulate(x),
the gated residual u, the MoE input m and the router input m', then the MoE
sub-layer with the output u + g_m y.  Cases: both attention cores, three head
sizes, samples ragged against the query blocks and GEMM tiles, the three
attention policies, a shared expert, the widest block (D 2560), the
full-size D 768 block, zero gates (exact pass-through), and a sampler loop
whose next input is the Eq. 1 update of the stack's output.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_harness import run_trajectory  # noqa: E402
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


def drift(x0, rng, n, sigma):
    xs = [x0]
    for _ in range(1, n):
        xs.append((xs[-1] + sigma * rng.standard_normal(x0.shape)).astype(np.float32))
    return [W.round_to_bf16(x) for x in xs]


def make_adaln_stack(M, T, D, H, E, k, F, L=1, S=0, n_shared=0, seed=0, wscale=0.05, ada_scale=0.05, **cfg_kw):
    ws = []
    for l in range(L):
        w, _, _ = W.tiny_layer(500 + 10 * seed + l, T, D, E, k, F, n_shared=n_shared, dtype="bf16",
                               bias=n_shared > 0, wscale=wscale)
        w.update(W.tiny_attn(500 + 10 * seed + l, D, dtype="bf16", wscale=wscale))
        w.update(W.tiny_adaln(500 + 10 * seed + l, D, dtype="bf16", wscale=ada_scale))
        ws.append(w)
    cfg = M.moeca_config_default(n_layers=L, hidden=D, ffn=F, n_experts=E, top_k=k, n_shared=n_shared,
                                 max_tokens=cfg_kw.pop("max_tokens", T), dtype=M.MOECA_BF16,
                                 n_heads=H, seq_len=S, adaln=1, keep_route_in=1, **cfg_kw)
    return M.Stack(cfg, ws), cfg, ws


@pytest.mark.parametrize("D,H,S,T,impl", [(256, 4, 200, 400, 2), (384, 4, 136, 272, 1), (576, 8, 104, 312, 1),
                                          (384, 3, 264, 528, 2)])
def test_sync_adaln_blocks(M, D, H, S, T, impl):
    """Heads of 64, 72 and 128 channels, ragged samples, two layers, a full
    step every 3 steps, the conditioning changing every step."""
    st, cfg, ws = make_adaln_stack(M, T, D, H, 8, 2, 256, L=2, S=S, seed=D + H, tau0=0.72, refresh_period=3,
                                   attn_impl=impl)
    rng = np.random.default_rng(D + H)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 5, 0.08)
    conds = W.conditioning(D + H, T // S, D, 5)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=conds)
    cache_rows = rep.attn_rows - 2 * 2 * T          # full steps 0 and 3, two layers
    assert rep.reused > 0 and rep.recomputed > 0
    assert 0 < cache_rows < 2 * 3 * T, rep
    assert st.stats()["attn_recomputed"] == rep.attn_rows
    st.close()


@pytest.mark.parametrize("policy", [1, 2])
def test_stale_and_full_policies(M, policy):
    T, D, H, S = 256, 256, 4, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 8, 2, 256, L=2, S=S, seed=7, tau0=0.72, attn_policy=policy)
    rng = np.random.default_rng(70 + policy)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.08)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=W.conditioning(7, T // S, D, 4))
    assert rep.attn_rows == (2 * 4 * T if policy == 2 else 2 * T)
    st.close()


def test_shared_expert_block(M):
    T, D, H, S = 256, 256, 4, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 4, 2, 256, L=1, S=S, n_shared=1, seed=8, tau0=0.72)
    rng = np.random.default_rng(80)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.08)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=W.conditioning(8, T // S, D, 4))
    assert rep.reused > 0 and rep.recomputed > 0
    st.close()


def test_token_reuse_copy_block(M):
    """Sec. 4.1's token-level reading in the AdaLN block: a token with an
    empty recompute set returns its stored ungated y^{t0}, and the current
    step's gate g_m applies to it (the conditioning changes every step)."""
    T, D, H, S = 256, 256, 4, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 4, 2, 256, L=2, S=S, n_shared=1, seed=12, tau0=0.95,
                                   token_reuse_policy=1)
    rng = np.random.default_rng(120)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.03)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=W.conditioning(12, T // S, D, 4))
    assert rep.tokens_copied > 0 and rep.recomputed > 0, rep.summary()
    st.close()


def test_wide_block(M):
    """D 2560 (20 heads of 128 channels), the widest row the AdaLN row kernel
    holds in registers (ten 16-byte chunks per lane)."""
    T, D, H, S = 256, 2560, 20, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 4, 2, 256, L=1, S=S, seed=9, tau0=0.72, wscale=0.02,
                                   ada_scale=0.02)
    rng = np.random.default_rng(90)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 3, 0.08)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=W.conditioning(9, T // S, D, 3))
    assert rep.layers_checked == 3
    st.close()


def test_full_size_d768_block(M):
    """The 12-head D 768 block of the 256px workloads: 8 samples of 256
    tokens, E 16, top-2, F 3072; one full step and two cache steps."""
    T, D, H, S, E, k, F = 2048, 768, 12, 256, 16, 2, 3072
    st, cfg, ws = make_adaln_stack(M, T, D, H, E, k, F, L=1, S=S, seed=11, tau0=0.7, wscale=0.02,
                                   ada_scale=0.02)
    rng = np.random.default_rng(110)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 3, 0.05)
    rep, _ = run_trajectory(st, cfg, ws, xs, conds=W.conditioning(11, T // S, D, 3))
    assert rep.reused > 0 and rep.recomputed > 0
    st.close()


def test_zero_gates_pass_the_input_through(M):
    """gate_a = gate_m = 0: u = bf16(x + 0 a) = x and out = bf16(u + 0 y) = x
    bit for bit, on full and cache steps."""
    T, D, H, S = 256, 256, 4, 128
    ws = []
    w, _, _ = W.tiny_layer(600, T, D, 8, 2, 256, dtype="bf16", wscale=0.05)
    w.update(W.tiny_attn(600, D, dtype="bf16", wscale=0.05))
    w.update(W.tiny_adaln(600, D, dtype="bf16", wscale=0.05))
    for j in (2, 5):
        w["w_ada"][j * D:(j + 1) * D] = 0
        w["b_ada"][j * D:(j + 1) * D] = 0
    ws.append(w)
    cfg = M.moeca_config_default(n_layers=1, hidden=D, ffn=256, n_experts=8, top_k=2, max_tokens=T,
                                 dtype=M.MOECA_BF16, n_heads=H, seq_len=S, adaln=1, tau0=0.72)
    st = M.Stack(cfg, ws)
    rng = np.random.default_rng(600)
    conds = W.conditioning(600, T // S, D, 3)
    for t in range(3):
        x = torch.from_numpy(W.round_to_bf16(rng.standard_normal((T, D)).astype(np.float32))).cuda().bfloat16()
        out = st.step(x, t, cond=torch.from_numpy(conds[t]).cuda())
        torch.cuda.synchronize()
        assert torch.equal(out, x)
    assert st.stats()["device_status"] == 0
    st.close()


def test_missing_conditioning_is_an_error(M):
    T, D, H, S = 256, 256, 4, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 8, 2, 256, S=S, seed=12)
    x = torch.zeros((T, D), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(M.MoecaError) as ei:
        st.step(x, 0)
    assert ei.value.status == M.MOECA_ERR_INVALID_ARG
    st.close()


@pytest.mark.parametrize("eps_dtype", ["bf16", "f32"])
def test_ddpm_step_matches_oracle(M, eps_dtype):
    """Eq. 1 on the GPU against the float64 oracle, every step of a 50-step
    schedule, with and without noise; x_next is x_prev in eps's dtype."""
    n = 8 * 1237
    rng = np.random.default_rng(5)
    dt = torch.bfloat16 if eps_dtype == "bf16" else torch.float32
    _, alpha, abar, beta = M.moeca_ddpm_schedule(50)
    for j in (49, 25, 1, 0):
        x = torch.from_numpy(rng.standard_normal(n).astype(np.float32)).cuda()
        eps = torch.from_numpy(rng.standard_normal(n).astype(np.float32)).cuda().to(dt)
        z = torch.from_numpy(rng.standard_normal(n).astype(np.float32)).cuda()
        sigma = math.sqrt(beta[j]) if j > 0 else 0.0
        x_next = torch.empty(n, dtype=dt, device="cuda")
        xp = M.ddpm_step(x, eps, alpha[j], abar[j], sigma, z=z if sigma else None, x_next=x_next)
        torch.cuda.synchronize()
        want = O.ddpm_step(x.cpu().numpy(), eps.float().cpu().numpy(), z.cpu().numpy() if sigma else 0.0,
                           alpha[j], abar[j], sigma)
        got = xp.cpu().numpy().astype(np.float64)
        np.testing.assert_allclose(got, want, rtol=2e-6, atol=2e-6 * np.abs(want).max())
        assert torch.equal(x_next, xp.to(dt))


def test_sampler_loop_feeds_the_stack(M):
    """Four steps of a 50-step reverse process: the AdaLN stack's output is
    eps, Eq. 1 (on the GPU, checked against the oracle on the GPU's inputs)
    gives the next input.  Every stack step is checked layer by layer."""
    T, D, H, S = 256, 256, 4, 128
    st, cfg, ws = make_adaln_stack(M, T, D, H, 8, 2, 256, L=2, S=S, seed=13, tau0=0.72)
    _, alpha, abar, beta = M.moeca_ddpm_schedule(50)
    rng = np.random.default_rng(130)
    x_t = torch.from_numpy(rng.standard_normal((T, D)).astype(np.float32)).cuda()
    conds = W.conditioning(13, T // S, D, 4)
    state = {"x": x_t}

    def next_input(t, eps):
        j = 49 - (t - 1)
        z = torch.from_numpy(rng.standard_normal((T, D)).astype(np.float32)).cuda()
        x_next = torch.empty((T, D), dtype=torch.bfloat16, device="cuda")
        xp = M.ddpm_step(state["x"], eps, alpha[j], abar[j], math.sqrt(beta[j]), z=z, x_next=x_next)
        torch.cuda.synchronize()
        want = O.ddpm_step(state["x"].cpu().numpy(), eps.float().cpu().numpy(), z.cpu().numpy(), alpha[j],
                           abar[j], math.sqrt(beta[j]))
        np.testing.assert_allclose(xp.cpu().numpy(), want, rtol=2e-6, atol=2e-6 * np.abs(want).max())
        state["x"] = xp
        return x_next.float().cpu().numpy()

    x0 = W.round_to_bf16(x_t.cpu().numpy())
    rep, _ = run_trajectory(st, cfg, ws, [x0], conds=conds, next_input=next_input, n_steps=4)
    assert rep.steps == 4 and rep.layers_checked == 8
    st.close()
