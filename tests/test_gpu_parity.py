"""GPU vs oracle parity, through the C ABI (marked gpu).

Every layer of every step is checked stage by stage against the oracle (see
gpu_harness).  Cases span several GEMM tiles (128 rows) and router / select
blocks with ragged tails, the fp32 debug path, the tensor-core and the SIMT
bf16 paths, a shared expert with skewed routing, the fine-grained 64-expert
top-8 shape, each reading switch, and the degenerate cases.
"""
import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

from gpu_harness import np_of, rel_l2, run_trajectory  # noqa: E402
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


def drift(x0, rng, n, sigma, bf16):
    xs = [x0]
    for _ in range(1, n):
        xs.append((xs[-1] + sigma * rng.standard_normal(x0.shape)).astype(np.float32))
    return [W.round_to_bf16(x) for x in xs] if bf16 else xs


def make_stack(M, T, D, E, k, F, L=1, S=0, bf16=True, seed=0, bias=False, wscale=0.05, **cfg_kw):
    ws = []
    for l in range(L):
        w, _, _ = W.tiny_layer(100 * seed + l, T, D, E, k, F, n_shared=S, dtype="bf16" if bf16 else "f32",
                               bias=bias, wscale=wscale)
        ws.append(w)
    cfg = M.moeca_config_default(n_layers=L, hidden=D, ffn=F, n_experts=E, top_k=k, n_shared=S,
                                 max_tokens=cfg_kw.pop("max_tokens", T),
                                 dtype=M.MOECA_BF16 if bf16 else M.MOECA_F32, **cfg_kw)
    return M.Stack(cfg, ws), cfg, ws


def test_fp32_workload_full_size(M):
    """The fp32 single-layer workload at full size: D 384, E 8, top-2, F 1536, T 512, 4 steps."""
    wl = W.workload(1)
    w = W.make_layer_weights(wl, 0)
    cfg = M.moeca_config_default(n_layers=1, hidden=wl.hidden, ffn=wl.ffn, n_experts=wl.n_experts,
                                 top_k=wl.top_k, max_tokens=wl.n_tokens, dtype=M.MOECA_F32, tau0=0.572)
    st = M.Stack(cfg, [w])
    xs = list(W.trajectory(wl))
    rep, out = run_trajectory(st, cfg, [w], xs, bf16=False)
    assert rep.reused > 0 and rep.recomputed > 0 and rep.unmatched > 0
    # Free-running: the whole trajectory in the oracle alone.
    ost = O.Stack([w], O.Params(top_k=2, tau0=0.572), wl.hidden, wl.n_experts)
    for t, x in enumerate(xs):
        o_out, infos = ost.step(x, t)
    assert rel_l2(np_of(out), o_out) <= 1e-5
    st.close()


@pytest.mark.parametrize("impl", ["tc", "simt"])
def test_bf16_stack_ragged(M, impl):
    """3 layers, T = 300 (ragged for 128-row tiles and 16/128-token blocks), refresh every 3."""
    T, D, E, k, F = 300, 256, 8, 2, 512
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=3, seed=1, tau0=0.75, refresh_period=3,
                             ffn_impl=M.MOECA_FFN_AUTO if impl == "tc" else M.MOECA_FFN_SIMT)
    rng = np.random.default_rng(11)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 5, 0.08, True)
    rep, _ = run_trajectory(st, cfg, ws, xs)
    assert rep.reused > 0 and rep.recomputed > 0 and rep.unmatched > 0, rep
    st.close()


def test_bf16_shared_expert_skewed(M):
    """One shared expert under the synchronized rule, 4 experts with a skewed router bias."""
    T, D, E, k, F = 260, 192, 4, 2, 320
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, S=1, seed=2, bias=True, tau0=0.7)
    rng = np.random.default_rng(12)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
    rep, _ = run_trajectory(st, cfg, ws, xs)
    stats = st.stats()
    assert 0 < stats["shared_recomputed"] < T * 2 * 4
    assert rep.reused > 0
    st.close()


def test_bf16_fine_grained_64_experts_top8(M):
    T, D, E, k, F = 257, 128, 64, 8, 128
    st, cfg, ws = make_stack(M, T, D, E, k, F, seed=3, tau0=0.25, lambda2=0.3)
    rng = np.random.default_rng(13)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
    rep, _ = run_trajectory(st, cfg, ws, xs)
    assert rep.reused > 0 and rep.recomputed > 0
    st.close()


@pytest.mark.parametrize("k,impl", [(3, "simt"), (4, "simt"), (4, "tc")])
def test_bf16_top3_top4(M, k, impl):
    """The kernels' middle top-k bound (k <= 4): the separate router / select /
    compact launches (the SIMT FFN takes them), and the fused preparation
    kernel.  The tau0 values give both reused and recomputed branches in the
    oracle on these inputs."""
    T, D, E, F = 233, 128, 16, 192
    kw = {"ffn_impl": M.MOECA_FFN_SIMT} if impl == "simt" else {}
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, seed=21 + k, tau0={3: 0.4, 4: 0.3}[k], **kw)
    rng = np.random.default_rng(60 + k)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
    rep, _ = run_trajectory(st, cfg, ws, xs)
    assert rep.reused > 0 and rep.recomputed > 0
    st.close()


@pytest.mark.parametrize("switch", [
    dict(entropy_norm=1), dict(reused_meta_policy=1), dict(shared_policy=1, n_shared=1),
    dict(gelu_tanh=0), dict(renorm_topk=0, tau0=0.45),
    # Table 5's score-signal subsets and token-level granularity (Sec. 3)
    dict(score_terms=1, tau0=0.55), dict(score_terms=2, tau0=0.05), dict(score_terms=4, tau0=0.25),
    dict(score_terms=3, tau0=0.6), dict(score_terms=6, tau0=0.3), dict(granularity=1, tau0=0.9),
    dict(granularity=1, score_terms=5, tau0=0.8),
    # Sec. 4.1's token-level reading: R_i empty => y^{t0} returned unchanged
    dict(token_reuse_policy=1, tau0=0.9), dict(token_reuse_policy=1, n_shared=1, tau0=1.0),
    dict(token_reuse_policy=1, granularity=1, tau0=0.95)])
def test_reading_switches(M, switch):
    sw = dict(switch)
    S = sw.pop("n_shared", 0)
    T, D, E, k, F = 140, 128, 8, 2, 192
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=1, S=S, seed=4, **({"tau0": 0.75} | sw))
    rng = np.random.default_rng(14)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
    rep, _ = run_trajectory(st, cfg, ws, xs)
    if sw.get("token_reuse_policy"):
        assert rep.tokens_copied > 0 and rep.recomputed > 0, rep.summary()
    st.close()


@pytest.mark.parametrize("bf16", [False, True])
def test_token_reuse_copy_multi_layer(M, bf16):
    """The copy reading on the fp32 separate-kernel path and on the bf16
    fused path, three layers, tokens reused for several steps in a row: the
    returned y must be the one stored when the token last computed."""
    T, D, E, k, F = 193, 128, 8, 2, 256
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=3, bf16=bf16, seed=9, tau0=0.95, token_reuse_policy=1,
                             refresh_period=5)
    rng = np.random.default_rng(19)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 6, 0.03, bf16)
    rep, out = run_trajectory(st, cfg, ws, xs, bf16=bf16)
    assert rep.tokens_copied > T and rep.recomputed > 0, rep.summary()
    st.close()


def test_fp32_reading_switches_and_k_equals_e(M):
    T, D, E, k, F = 90, 64, 4, 4, 96
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, bf16=False, seed=5, tau0=0.3, entropy_norm=1,
                             reused_meta_policy=1)
    rng = np.random.default_rng(15)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.1, False)
    rep, _ = run_trajectory(st, cfg, ws, xs, bf16=False)
    assert rep.unmatched == 0, "with k = E every branch is matched"
    st.close()


def test_token_count_changes_single_token_and_empty_step(M):
    T, D, E, k, F = 200, 128, 8, 2, 128
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, seed=6, tau0=0.75, max_tokens=200)
    rng = np.random.default_rng(16)
    a = drift(rng.standard_normal((200, D)).astype(np.float32), rng, 2, 0.05, True)
    b = drift(rng.standard_normal((1, D)).astype(np.float32), rng, 2, 0.05, True)
    c = drift(rng.standard_normal((77, D)).astype(np.float32), rng, 2, 0.05, True)
    flags = []
    run_trajectory(st, cfg, ws, a + b + c, refresh_flags=flags)
    assert flags == [True, False, True, False, True, False]
    x = torch.zeros((0, D), dtype=torch.bfloat16, device="cuda")
    st.step(x, 9)  # T = 0 is a no-op
    st.close()


def test_forced_refresh_and_tau_override(M):
    T, D, E, k, F = 150, 128, 8, 2, 128
    st, cfg, ws = make_stack(M, T, D, E, k, F, seed=7, tau0=0.75)
    rng = np.random.default_rng(17)
    xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
    flags = []
    run_trajectory(st, cfg, ws, xs, refresh_flags=flags, forces=[False, False, True, False])
    assert flags == [True, False, True, False]
    # tau0 = -inf per step: every branch recomputed.
    M.moeca_reset_stats(st.handle)
    xd = torch.from_numpy(xs[-1]).cuda().to(torch.bfloat16)
    st.step(xd, 4, tau0=-math.inf)
    s = st.stats()
    assert s["reused"] == 0 and s["recomputed"] == T * k
    st.close()


def test_everything_reused_gives_bitwise_identical_output(M):
    T, D, E, k, F = 200, 128, 8, 2, 256
    st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, S=1, seed=8, tau0=math.inf)
    x = torch.from_numpy(W.round_to_bf16(np.random.default_rng(18).standard_normal((T, D)).astype(np.float32))).cuda().to(torch.bfloat16)
    o1 = st.step(x, 0).clone()
    o2 = st.step(x, 1).clone()
    o3 = st.step(x, 2).clone()
    assert torch.equal(o1, o2) and torch.equal(o1, o3)
    s = st.stats()
    assert s["reused"] == 2 * 2 * T * k and s["tokens_fully_reused"] == 2 * 2 * T
    assert s["shared_recomputed"] == 2 * T  # only on the full step, in both layers
    st.close()


def test_deterministic_across_handles(M):
    T, D, E, k, F = 300, 128, 16, 2, 256
    outs = []
    for _ in range(2):
        st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, seed=9, tau0=0.75)
        rng = np.random.default_rng(19)
        xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 3, 0.05, True)
        for t, x in enumerate(xs):
            o = st.step(torch.from_numpy(x).cuda().to(torch.bfloat16), t)
        tr = st.get_trace(1, T)
        outs.append((o.clone(), {kk: v.clone() for kk, v in tr.items()}, st.stats()))
        st.close()
    assert torch.equal(outs[0][0], outs[1][0])
    for kk in outs[0][1]:
        assert torch.equal(outs[0][1][kk], outs[1][1][kk]), kk
    assert outs[0][2] == outs[1][2]


def test_tc_and_simt_agree(M):
    T, D, E, k, F = 384, 256, 8, 2, 384
    res = []
    for impl in (M.MOECA_FFN_AUTO, M.MOECA_FFN_SIMT):
        st, cfg, ws = make_stack(M, T, D, E, k, F, seed=10, tau0=-math.inf, ffn_impl=impl)
        x = torch.from_numpy(W.round_to_bf16(np.random.default_rng(20).standard_normal((T, D)).astype(np.float32))).cuda().to(torch.bfloat16)
        res.append(np_of(st.step(x, 0)))
        st.close()
    assert rel_l2(res[0], res[1]) < 5e-3


@pytest.mark.parametrize("split", [2, 3])
def test_ffn_k_splits(M, split):
    """The second GEMM split along K (forced; 600 tokens, 16 m-tiles, phase 2
    in 64-wide tiles with 6 K stages): parity against the oracle over a
    two-layer trajectory, and the same bits on a second handle (the last
    split to arrive adds the parked tiles in split order, whichever arrives
    first)."""
    T, D, E, k, F = 600, 256, 8, 2, 768
    finals = []
    for run in range(2):
        st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, seed=12, tau0=0.75, ffn_split_k=split)
        rng = np.random.default_rng(120)
        xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
        if run == 0:
            rep, out = run_trajectory(st, cfg, ws, xs)
            assert rep.reused > 0 and rep.recomputed > 0, rep
        else:
            for t, x in enumerate(xs):
                out = st.step(torch.from_numpy(x).cuda().to(torch.bfloat16), t)
        torch.cuda.synchronize()
        finals.append(out.clone())
        st.close()
    assert torch.equal(finals[0], finals[1])


@pytest.mark.parametrize("shape", [
    dict(T=300, D=256, E=8, k=2, F=256, S=1, bf16=True),
    dict(T=257, D=128, E=16, k=8, F=128, S=0, bf16=True),
    dict(T=190, D=128, E=8, k=2, F=128, S=0, bf16=False)])
def test_staged_and_direct_combine_agree(M, shape):
    """The staged combine (rows brought into shared memory by bulk copies,
    two tokens in flight per warp) and the direct one give the same bits:
    outputs, cached norms and cache rows, over cache steps with reuse."""
    sh = dict(shape)
    bf16 = sh.pop("bf16")
    outs, states = [], []
    for direct in (0, 1):
        st, cfg, ws = make_stack(M, sh["T"], sh["D"], sh["E"], sh["k"], sh["F"], L=2, S=sh["S"], bf16=bf16,
                                 seed=31, bias=sh["S"] > 0, tau0=0.75 if sh["k"] == 2 else 0.25, combine_direct=direct)
        rng = np.random.default_rng(310)
        xs = drift(rng.standard_normal((sh["T"], sh["D"])).astype(np.float32), rng, 4, 0.05, bf16)
        dt = torch.bfloat16 if bf16 else torch.float32
        o = [st.step(torch.from_numpy(x).cuda().to(dt), t).clone() for t, x in enumerate(xs)]
        torch.cuda.synchronize()
        outs.append(o)
        states.append([st.get_state(l) for l in range(2)])
        assert st.stats()["reused"] > 0
        st.close()
    for a, b in zip(outs[0], outs[1]):
        assert torch.equal(a, b)
    for sa, sb in zip(states[0], states[1]):
        for key in ("cache_norm", "cache_h", "cache_e", "cache_w"):
            assert torch.equal(sa[key], sb[key]), key


def test_weight_prefetch_is_only_a_hint(M):
    """The preparation kernel's L2 prefetch of the routed W1 (none, the first
    1 MB of the 4 MB W1, and a cap above the whole W1) leaves every result
    bit unchanged: outputs, cached norms and cache rows, over cache steps
    with reuse."""
    T, D, E, k, F = 300, 256, 8, 2, 1024
    outs, states = [], []
    for mb in (0, 1, 4096):
        st, cfg, ws = make_stack(M, T, D, E, k, F, L=2, seed=33, tau0=0.75, weight_prefetch_mb=mb)
        rng = np.random.default_rng(330)
        xs = drift(rng.standard_normal((T, D)).astype(np.float32), rng, 4, 0.05, True)
        o = [st.step(torch.from_numpy(x).cuda().to(torch.bfloat16), t).clone() for t, x in enumerate(xs)]
        torch.cuda.synchronize()
        outs.append(o)
        states.append([st.get_state(l) for l in range(2)])
        assert st.stats()["reused"] > 0
        st.close()
    for other in (1, 2):
        for a, b in zip(outs[0], outs[other]):
            assert torch.equal(a, b)
        for sa, sb in zip(states[0], states[other]):
            for key in ("cache_norm", "cache_h", "cache_e", "cache_w"):
                assert torch.equal(sa[key], sb[key]), key
