"""The host-buffer step (moeca_step_host) against the device-buffer step, and
the measurement probes (marked gpu).

moeca_step_host uploads each input into double-buffered device staging on
its own stream, runs the same step and reads the output back on another
stream; its outputs must equal moeca_step's bit for bit on a twin handle,
across a change of token count and with an AdaLN stack's host-side
conditioning.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from paper_2606_15615_gb300 import workloads as W  # noqa: E402


@pytest.fixture(scope="module")
def M():
    if not torch.cuda.is_available():
        pytest.fail("a CUDA GPU is required for gpu-marked tests")
    from paper_2606_15615_gb300 import build
    build.build()
    from paper_2606_15615_gb300 import moeca
    return moeca


def _twins(M, cfg, ws):
    return M.Stack(cfg, ws), M.Stack(cfg, ws)


def test_host_step_equals_device_step(M):
    T, D, E, k, F, L = 300, 128, 8, 2, 256, 2
    ws = [W.tiny_layer(700 + l, T, D, E, k, F, dtype="bf16", wscale=0.05)[0] for l in range(L)]
    cfg = M.moeca_config_default(n_layers=L, hidden=D, ffn=F, n_experts=E, top_k=k, max_tokens=T,
                                 dtype=M.MOECA_BF16, tau0=0.75)
    dev_st, host_st = _twins(M, cfg, ws)
    rng = np.random.default_rng(70)
    Ts = [300, 300, 300, 211, 211, 211]
    x = rng.standard_normal((T, D)).astype(np.float32)
    xs = []
    for t, n in enumerate(Ts):
        x = x + 0.05 * rng.standard_normal((T, D)).astype(np.float32)
        xs.append(torch.from_numpy(W.round_to_bf16(x[:n])).to(torch.bfloat16).pin_memory())
    outs_host = [torch.empty_like(v).pin_memory() for v in xs]
    stream = torch.cuda.current_stream().cuda_stream
    for t, (xh, oh) in enumerate(zip(xs, outs_host)):
        M.moeca_step_host(host_st.handle, xh.data_ptr(), oh.data_ptr(), xh.shape[0], t, stream=stream)
    M.moeca_host_join(host_st.handle, stream)
    torch.cuda.current_stream().synchronize()
    for t, (xh, oh) in enumerate(zip(xs, outs_host)):
        ref = dev_st.step(xh.cuda(), t)
        torch.cuda.synchronize()
        assert torch.equal(ref.cpu(), oh), f"step {t}"
    assert host_st.stats()["reused"] == dev_st.stats()["reused"] > 0
    dev_st.close()
    host_st.close()


def test_host_step_adaln_conditioning(M):
    T, D, H, S, E, k, F = 256, 128, 2, 128, 4, 2, 256
    w, _, _ = W.tiny_layer(710, T, D, E, k, F, dtype="bf16", wscale=0.05)
    w.update(W.tiny_attn(710, D, dtype="bf16", wscale=0.05))
    w.update(W.tiny_adaln(710, D, dtype="bf16", wscale=0.05))
    cfg = M.moeca_config_default(n_layers=1, hidden=D, ffn=F, n_experts=E, top_k=k, max_tokens=T,
                                 dtype=M.MOECA_BF16, tau0=0.75, n_heads=H, seq_len=S, adaln=1)
    dev_st, host_st = _twins(M, cfg, [w])
    rng = np.random.default_rng(71)
    conds = W.conditioning(710, T // S, D, 4)
    x = rng.standard_normal((T, D)).astype(np.float32)
    stream = torch.cuda.current_stream().cuda_stream
    for t in range(4):
        x = x + 0.05 * rng.standard_normal((T, D)).astype(np.float32)
        xh = torch.from_numpy(W.round_to_bf16(x)).to(torch.bfloat16).pin_memory()
        ch = torch.from_numpy(np.ascontiguousarray(conds[t], np.float32)).pin_memory()
        oh = torch.empty_like(xh).pin_memory()
        M.moeca_step_host(host_st.handle, xh.data_ptr(), oh.data_ptr(), T, t, stream=stream,
                          cond_host_ptr=ch.data_ptr())
        M.moeca_host_join(host_st.handle, stream)
        torch.cuda.current_stream().synchronize()
        ref = dev_st.step(xh.cuda(), t, cond=ch.cuda())
        torch.cuda.synchronize()
        assert torch.equal(ref.cpu(), oh), f"step {t}"
    dev_st.close()
    host_st.close()


def test_ffma_probe(M):
    tf, ms = M.moeca_probe_ffma(0)
    # 152 SMs x 128 FP32 lanes x 2 flops at up to 2.07 GHz is 80.5 TFLOP/s.
    assert 10.0 < tf < 100.0 and ms > 0.0, (tf, ms)


def test_stream_probe(M):
    # 4096 tokens x (2 rows read + 1 written) of 2304 B: 28 MB in, 9 MB out.
    gbs, us = M.moeca_probe_stream(0, 4096, 2, 2304, reps=5)
    assert 100.0 < gbs < 20000.0 and us > 0.0, (gbs, us)
    assert abs(gbs - 4096 * 3 * 2304 / (us * 1e-6) / 1e9) < 1e-6 * gbs
    with pytest.raises(M.MoecaError):
        M.moeca_probe_stream(0, 4096, 11, 2304)
    with pytest.raises(M.MoecaError):
        M.moeca_probe_stream(0, 4096, 2, 2300)
