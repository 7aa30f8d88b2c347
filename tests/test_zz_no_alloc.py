"""The allocation-free router call, against the router inside moeca_step (marked gpu).

moeca_route_noalloc serves callers that cannot allocate device memory (a host
framework that owns all device memory, a fixed device-memory budget): it runs
one layer's router on the caller's buffers with scratch compiled into the
library.  Here its routing, gate weights, EMA statistic and thresholds must
match what a one-layer handle computes in moeca_step, on two calls in a row
(the second continues from the statistic the first left), within the same
tolerances as the other parity tests.  This file is collected last so that a
run stopping at the first failure has already run every other test.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_harness import (Report, assert_margins, check_gate_weights, count_route_margins, np_of,  # noqa: E402
                         oracle_weights, params_of)
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


def _noalloc(M, cfg, x, wg, bg, ema, T):
    dev = x.device
    route_e = torch.empty((T, cfg.top_k), dtype=torch.int32, device=dev)
    route_w = torch.empty((T, cfg.top_k), dtype=torch.float32, device=dev)
    tau = torch.empty((cfg.n_experts,), dtype=torch.float32, device=dev)
    a = M.moeca_route_args(
        dtype=cfg.dtype, n_tokens=T, hidden=cfg.hidden, n_experts=cfg.n_experts, top_k=cfg.top_k,
        renorm_topk=cfg.renorm_topk, entropy_norm=cfg.entropy_norm, beta=cfg.beta, tau0=cfg.tau0,
        alpha=cfg.alpha, x=x.data_ptr(), w_gate=wg.data_ptr(), b_gate=bg.data_ptr() if bg is not None else None,
        ema=ema.data_ptr(), route_e=route_e.data_ptr(), route_w=route_w.data_ptr(), tau=tau.data_ptr())
    M.moeca_route_noalloc(a, torch.cuda.current_stream().cuda_stream)
    return route_e, route_w, tau


@pytest.mark.parametrize("bf16", [True, False])
def test_noalloc_router_matches_moeca_step_twice(M, bf16):
    T, D, E, k, F = 300, 256, 16, 2, 128
    w, x0, rng = W.tiny_layer(31, T, D, E, k, F, dtype="bf16" if bf16 else "f32", bias=True, wscale=0.05)
    cfg = M.moeca_config_default(n_layers=1, hidden=D, ffn=F, n_experts=E, top_k=k, max_tokens=T,
                                 dtype=M.MOECA_BF16 if bf16 else M.MOECA_F32, tau0=0.75)
    stack = M.Stack(cfg, [w])
    dt = torch.bfloat16 if bf16 else torch.float32
    wg = torch.from_numpy(w["w_gate"]).cuda().to(dt)
    bg = torch.from_numpy(w["b_gate"]).cuda()
    ema = torch.zeros((T, E), dtype=torch.float32, device="cuda")
    x1 = x0 + 0.05 * rng.standard_normal(x0.shape).astype(np.float32)
    for t, xn in enumerate([x0, x1]):
        if bf16:
            xn = W.round_to_bf16(xn)
        x = torch.from_numpy(np.ascontiguousarray(xn, np.float32)).cuda().to(dt)
        stack.step(x, t)
        tr = stack.get_trace(0, T)
        st = stack.get_state(0)
        e, rw, tau = _noalloc(M, cfg, x, wg, bg, ema, T)
        torch.cuda.synchronize()
        assert torch.equal(e, tr["route_e"])
        assert np.allclose(np_of(rw), np_of(tr["route_w"]), rtol=0, atol=2e-6)
        assert np.allclose(np_of(ema), np_of(st["ema"]), rtol=2e-6, atol=1e-7)
        assert np.allclose(np_of(tau), np_of(tr["tau"]), rtol=1e-5, atol=1e-6)
    stack.close()


@pytest.mark.parametrize("D,bf16", [(1152, True), (1536, True), (1152, False)])
def test_noalloc_wide_gate_router_against_oracle(M, D, bf16):
    """64 experts, top-8, 300 tokens (a ragged last block), two calls in a row,
    against the oracle: the ids outside near ties, the gate weights, the EMA
    statistic (Eq. 10) and the thresholds (Eq. 11-12).  The shapes take the
    router's wide-gate forms: 32-token blocks with the gate matrix and the
    token rows in shared memory together (D 1152, bf16), 16-token blocks with
    the token rows read through L1 (D 1536), and the fp32 form."""
    T, E, k = 300, 64, 8
    w, x0, rng = W.tiny_layer(41, T, D, E, k, 64, dtype="bf16" if bf16 else "f32", bias=True, wscale=0.05)
    cfg = M.moeca_config_default(n_layers=1, hidden=D, ffn=64, n_experts=E, top_k=k, max_tokens=T,
                                 dtype=M.MOECA_BF16 if bf16 else M.MOECA_F32, tau0=0.75)
    prm = params_of(cfg)
    dt = torch.bfloat16 if bf16 else torch.float32
    wg = torch.from_numpy(w["w_gate"]).cuda().to(dt)
    bg = torch.from_numpy(w["b_gate"]).cuda()
    wo = oracle_weights({"w_gate": w["w_gate"], "b_gate": w["b_gate"]})
    ema = torch.zeros((T, E), dtype=torch.float32, device="cuda")
    rep = Report()
    C_pre = np.zeros((E, T))
    x1 = x0 + 0.05 * rng.standard_normal(x0.shape).astype(np.float32)
    for xn in (x0, x1):
        if bf16:
            xn = W.round_to_bf16(xn)
        x = torch.from_numpy(np.ascontiguousarray(xn, np.float32)).cuda().to(dt)
        e, rw, tau = _noalloc(M, cfg, x, wg, bg, ema, T)
        torch.cuda.synchronize()
        e_g = np_of(e).astype(np.int64)
        w_g = np_of(rw).astype(np.float64)
        e_o, w_o, ok, cond = count_route_margins(rep, np_of(x).astype(np.float64), wo, k, bool(cfg.renorm_topk), e_g)
        bad = np.nonzero(ok & (e_o != e_g).any(axis=1))[0]
        assert len(bad) == 0, f"top-k ids differ on {len(bad)} tokens, e.g. {bad[:5]}"
        check_gate_weights(w_g[ok], w_o[ok], cond[ok])
        C_g = np_of(ema).astype(np.float64).T
        C_o = O.ema_update(C_pre, e_g, prm.beta)
        assert np.allclose(C_g, C_o, rtol=2e-6, atol=1e-7), f"EMA: max err {np.abs(C_g - C_o).max()}"
        tau_o = O.expert_threshold(O.normalized_entropy(C_g, prm.entropy_norm), prm.tau0, prm.alpha)
        tau_g = np_of(tau).astype(np.float64)
        assert np.allclose(tau_g, tau_o, rtol=1e-5, atol=1e-6), f"tau: max err {np.abs(tau_g - tau_o).max()}"
        C_pre = C_g
    assert_margins(rep)


def test_noalloc_rejects_sizes_beyond_its_scratch(M):
    E = 64
    T = 16 * (32768 // E) + 1  # one 16-token block more than the scratch holds
    a = M.moeca_route_args(dtype=M.MOECA_BF16, n_tokens=T, hidden=64, n_experts=E, top_k=2, renorm_topk=1,
                           entropy_norm=0, beta=0.65, tau0=0.8, alpha=0.6, x=256, w_gate=256, b_gate=None,
                           ema=256, route_e=256, route_w=256, tau=256)
    with pytest.raises(M.MoecaError) as ei:
        M.moeca_route_noalloc(a)
    assert ei.value.status == -2  # MOECA_ERR_UNSUPPORTED, nothing launched
    a.n_tokens = 0
    with pytest.raises(M.MoecaError) as ei:
        M.moeca_route_noalloc(a)
    assert ei.value.status == -1
