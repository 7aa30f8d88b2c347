"""The C-ABI library builds, loads without a GPU and exports what the header declares."""
import ctypes

import pytest

from paper_2606_15615_gb300 import build


@pytest.fixture(scope="module")
def lib():
    build.build()
    from paper_2606_15615_gb300 import moeca
    return moeca


def test_every_declared_function_is_exported(lib):
    names = lib.header_functions()
    assert len(names) >= 14
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in names if not hasattr(so, n)]
    assert not missing, missing


def test_status_strings_and_defaults(lib):
    assert lib.moeca_status_string(0) == "ok"
    assert lib.moeca_status_string(-1) == "invalid argument"
    assert lib.moeca_status_string(-6) == "device wait timed out"
    cfg = lib.moeca_config_default()
    assert (cfg.lambda1, cfg.lambda2) == (1.0, 0.5)
    assert abs(cfg.tau0 - 0.8) < 1e-7 and abs(cfg.alpha - 0.6) < 1e-7 and abs(cfg.beta - 0.65) < 1e-7
    assert cfg.renorm_topk == 1 and cfg.gelu_tanh == 1 and cfg.dtype == lib.MOECA_BF16
    assert cfg.score_terms == 7 and cfg.granularity == 0
    assert (cfg.n_heads, cfg.seq_len, cfg.attn_policy) == (0, 0, lib.ATTN_SYNC)
    assert cfg.combine_direct == 1 and cfg.weight_prefetch_mb == 16
    # The Python mirror of moeca_config ends at the header's last field.
    assert ctypes.sizeof(lib.moeca_config) == lib.moeca_config.weight_prefetch_mb.offset + 4


def test_host_validation_needs_no_gpu(lib):
    L = lib.LIB
    h = ctypes.c_void_p()
    assert L.moeca_create(None, None, 0, ctypes.byref(h)) == -1
    assert b"NULL" in L.moeca_last_error(None)
    cfg = lib.moeca_config_default(n_layers=1, hidden=64, ffn=64, n_experts=4, top_k=5, max_tokens=8)
    w = (lib.moeca_layer_weights * 1)()
    assert L.moeca_create(ctypes.byref(cfg), w, 0, ctypes.byref(h)) == -1  # top_k > E
    cfg.top_k = 2
    cfg.alpha = 1.0
    assert L.moeca_create(ctypes.byref(cfg), w, 0, ctypes.byref(h)) == -1  # alpha outside [0, 1)
    cfg.alpha = 0.6
    for bad in (dict(score_terms=0), dict(score_terms=8), dict(granularity=2)):
        c2 = lib.moeca_config_default(n_layers=1, hidden=64, ffn=64, n_experts=4, top_k=2, max_tokens=8, **bad)
        assert L.moeca_create(ctypes.byref(c2), w, 0, ctypes.byref(h)) == -1
        assert b"score_terms" in L.moeca_last_error(None)
    for bad in (-1, 4097):
        c2 = lib.moeca_config_default(n_layers=1, hidden=64, ffn=64, n_experts=4, top_k=2, max_tokens=8,
                                      weight_prefetch_mb=bad)
        assert L.moeca_create(ctypes.byref(c2), w, 0, ctypes.byref(h)) == -1
        assert b"weight_prefetch_mb" in L.moeca_last_error(None)
    assert L.moeca_create(ctypes.byref(cfg), w, 0, ctypes.byref(h)) == -1  # NULL weights
    cfg.hidden = 60
    w[0].w_gate = w[0].w1 = w[0].w2 = 4096
    assert L.moeca_create(ctypes.byref(cfg), w, 0, ctypes.byref(h)) == -2  # hidden not a multiple of 8
    assert L.moeca_step(None, None, None, None, None) == -1
    assert L.moeca_destroy(None) == 0


def test_attention_config_validation_needs_no_gpu(lib):
    """DiT-MoE block settings are checked before any device call."""
    L = lib.LIB
    h = ctypes.c_void_p()
    w = (lib.moeca_layer_weights * 1)()
    w[0].w_gate = w[0].w1 = w[0].w2 = 4096

    def create(**kw):
        base = dict(n_layers=1, hidden=768, ffn=256, n_experts=4, top_k=2, max_tokens=8)
        base.update(kw)
        c = lib.moeca_config_default(**base)
        return L.moeca_create(ctypes.byref(c), w, 0, ctypes.byref(h))

    for bad in (dict(n_heads=-1), dict(seq_len=-2), dict(attn_policy=3), dict(n_heads=12, attn_policy=-1)):
        assert create(**bad) == lib.MOECA_ERR_INVALID_ARG, bad
    assert create(n_heads=12, dtype=lib.MOECA_F32) == lib.MOECA_ERR_UNSUPPORTED   # bf16 only
    assert create(n_heads=7) == lib.MOECA_ERR_UNSUPPORTED                      # 768 / 7 not a head size
    assert create(n_heads=24) == lib.MOECA_ERR_UNSUPPORTED                     # 32 channels per head
    assert create(n_heads=12) == lib.MOECA_ERR_INVALID_ARG                     # no attention weights
    assert b"attention weights" in L.moeca_last_error(None)


def test_adaln_config_validation_needs_no_gpu(lib):
    """AdaLN settings are checked before any device call."""
    L = lib.LIB
    h = ctypes.c_void_p()
    w = (lib.moeca_layer_weights * 1)()
    w[0].w_gate = w[0].w1 = w[0].w2 = w[0].w_qkv = w[0].w_o = 4096

    def create(**kw):
        base = dict(n_layers=1, hidden=768, ffn=256, n_experts=4, top_k=2, max_tokens=512)
        base.update(kw)
        c = lib.moeca_config_default(**base)
        return L.moeca_create(ctypes.byref(c), w, 0, ctypes.byref(h))

    cfg = lib.moeca_config_default()
    assert cfg.adaln == 0 and cfg.keep_route_in == 0 and abs(cfg.ln_eps - 1e-6) < 1e-12
    assert create(adaln=2, n_heads=12) == lib.MOECA_ERR_INVALID_ARG
    assert create(adaln=1) == lib.MOECA_ERR_UNSUPPORTED                     # AdaLN needs a DiT block
    assert create(adaln=1, n_heads=12, ln_eps=0.0) == lib.MOECA_ERR_INVALID_ARG
    # 512 one-token samples: 512 x 768 x 4 bytes of staged conditioning do not fit
    assert create(adaln=1, n_heads=12, seq_len=1) == lib.MOECA_ERR_UNSUPPORTED
    assert create(adaln=1, n_heads=12, seq_len=256) == lib.MOECA_ERR_INVALID_ARG  # no AdaLN weights
    assert b"AdaLN weights" in L.moeca_last_error(None)


def test_ddpm_schedule_matches_the_oracle(lib):
    """The library's Eq. 1 schedule (host code) against the oracle's."""
    import numpy as np
    from oracle import moeca_oracle as O
    for n in (2, 7, 50, 250, 1000):
        t, a, ab, b = lib.moeca_ddpm_schedule(n)
        to, ao, abo, bo = O.ddpm_schedule(n)
        assert np.array_equal(t, to)
        np.testing.assert_allclose(a, ao, rtol=1e-13)
        np.testing.assert_allclose(ab, abo, rtol=1e-13)
        np.testing.assert_allclose(b, bo, rtol=1e-9, atol=1e-15)
    for bad in ((1, 1000), (1001, 1000)):
        with pytest.raises(lib.MoecaError):
            lib.moeca_ddpm_schedule(*bad)
    args = lib.moeca_ddpm_args(n=12, eps_dtype=lib.MOECA_BF16, alpha=0.9, alpha_bar=0.5, sigma=0.1,
                               x_t=4096, eps=4096, z=4096, x_prev=4096)
    with pytest.raises(lib.MoecaError):          # n not a multiple of 8: refused before any launch
        lib.moeca_ddpm_step(args)
