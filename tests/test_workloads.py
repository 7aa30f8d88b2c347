"""The seeded input generators: determinism, shapes, bf16 rounding, router skew."""
import numpy as np
import torch

from paper_2606_15615_gb300 import workloads as W


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 3
    x[:4] = [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -0.0, 65504.0]  # ties both ways
    ours = W.round_to_bf16(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(ours.view(np.uint32), ref.view(np.uint32))
    assert np.array_equal(W.from_bf16_bits(W.bf16_bits(ours)), ours)


def test_weights_and_trajectory_are_seeded_and_shaped():
    wl = W.workload(2).scaled(batch=1, seq=64, n_layers=2, hidden=96, ffn=160)
    a = W.make_layer_weights(wl, 1)
    b = W.make_layer_weights(wl, 1)
    c = W.make_layer_weights(wl, 0)
    for key in ("w_gate", "w1", "w2"):
        assert np.array_equal(a[key], b[key]) and not np.array_equal(a[key], c[key])
        assert np.array_equal(W.round_to_bf16(a[key]), a[key])
    assert a["w1"].shape == (16, 160, 96) and a["w2"].shape == (16, 96, 160)
    assert abs(float(a["w1"].std()) - 0.02) < 1e-3
    t1 = list(W.trajectory(wl, 5))
    t2 = list(W.trajectory(wl, 5))
    assert len(t1) == 5 and all(np.array_equal(p, q) for p, q in zip(t1, t2))
    assert t1[0].shape == (64, 96)
    d1 = np.abs(t1[1] - t1[0]).mean()
    d4 = np.abs(t1[4] - t1[3]).mean()
    assert d4 < d1, "drift sigma decays along the trajectory"


def test_router_skew_bias_gives_4_2_1_1_loads():
    wl = W.workload(4).scaled(seq=20000)
    b = W._skew_bias(wl)
    s = 0.02 * np.sqrt(wl.hidden)
    rng = np.random.default_rng(1)
    z = rng.standard_normal((20000, 4)) * s + b
    top2 = np.argsort(-z, axis=1)[:, :2]
    load = np.bincount(top2.ravel(), minlength=4) / 20000
    np.testing.assert_allclose(load, [1.0, 0.5, 0.25, 0.25], atol=0.02)
