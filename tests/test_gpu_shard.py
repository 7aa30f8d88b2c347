"""Token-sharded steps (moeca_shard_begin / moeca_shard_next) on one GPU
(marked gpu).

Two rank handles each hold half of the batch; their per-layer exchange of
Eq. 11's entropy partials is done here by device copies between their
launches, which run one after the other on one stream (no kernel waits on
another).  Thresholds, decisions, row lists, cache state and outputs must be
bit-identical to a single handle stepping the whole batch with moeca_step.
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


def _stack(M, ws, T, D, E, k, F, S, **kw):
    cfg = M.moeca_config_default(n_layers=len(ws), hidden=D, ffn=F, n_experts=E, top_k=k, n_shared=S, max_tokens=T,
                                 dtype=M.MOECA_BF16, **kw)
    return M.Stack(cfg, ws)


def _emulated_sharded_step(M, ranks, xs_r, t, world, tau0=float("nan")):
    """One step of every rank: begin, then per layer the all-gather as copies."""
    n = xs_r[0].shape[0]
    nbytes = M.moeca_shard_exchange_bytes(ranks[0].handle, n)
    sends = [torch.zeros(nbytes, dtype=torch.uint8, device="cuda") for _ in ranks]
    recvs = [torch.zeros(world * nbytes, dtype=torch.uint8, device="cuda") for _ in ranks]
    outs = [torch.empty_like(x) for x in xs_r]
    sp = torch.cuda.current_stream().cuda_stream
    for r, st in enumerate(ranks):
        M.moeca_shard_begin(st.handle, xs_r[r].data_ptr(), outs[r].data_ptr(), n, t, r, world, sends[r].data_ptr(),
                            recvs[r].data_ptr(), tau0_override=tau0, stream=sp)
    while True:
        for recv in recvs:
            for r, send in enumerate(sends):
                recv[r * nbytes:(r + 1) * nbytes].copy_(send)
        done = [M.moeca_shard_next(st.handle, sp) for st in ranks]
        assert len(set(done)) == 1
        if done[0]:
            return outs


@pytest.mark.parametrize("case", [
    dict(T=256, D=256, E=8, k=2, F=256, S=0, L=3),
    dict(T=512, D=192, E=4, k=2, F=320, S=1, L=2, bias=True),
    dict(T=384, D=128, E=16, k=4, F=128, S=0, L=2, world=3)])
def test_sharded_equals_single_rank(M, case):
    c = dict(case)
    world = c.pop("world", 2)
    T, D, E, k, F, S, L = (c[key] for key in ("T", "D", "E", "k", "F", "S", "L"))
    ws = [W.tiny_layer(600 + l, T, D, E, k, F, n_shared=S, dtype="bf16", bias=c.get("bias", False),
                       wscale=0.05)[0] for l in range(L)]
    tau0 = 0.75 if k == 2 else 0.4
    full = _stack(M, ws, T, D, E, k, F, S, tau0=tau0, refresh_period=3)
    n = T // world
    ranks = [_stack(M, ws, n, D, E, k, F, S, tau0=tau0, refresh_period=3) for _ in range(world)]
    rng = np.random.default_rng(60)
    x = rng.standard_normal((T, D)).astype(np.float32)
    reused = 0
    for t in range(5):
        x = x + 0.05 * rng.standard_normal((T, D)).astype(np.float32)
        xb = torch.from_numpy(W.round_to_bf16(x)).cuda().to(torch.bfloat16)
        ref = full.step(xb, t)
        outs = _emulated_sharded_step(M, ranks, [xb[r * n:(r + 1) * n].contiguous() for r in range(world)], t,
                                      world)
        torch.cuda.synchronize()
        assert torch.equal(torch.cat(outs), ref), f"step {t}: outputs differ"
        for l in range(L):
            tr = full.get_trace(l, T)
            trs = [st.get_trace(l, n) for st in ranks]
            for r, tr_r in enumerate(trs):
                assert torch.equal(tr_r["tau"], tr["tau"]), f"step {t} layer {l} rank {r}: tau"
                for key in ("route_e", "route_w", "recompute", "slot", "matched", "token_any"):
                    assert torch.equal(tr_r[key], tr[key][r * n:(r + 1) * n]), (t, l, r, key)
            # Every group's rows: the ranks' lists in rank order, tokens shifted to global rows.
            cnt, off, lst = (tr[key].cpu().numpy() for key in ("counts", "offsets", "list"))
            for g in range(E + S):
                want = lst[off[g]:off[g] + cnt[g]]
                got = []
                for r, tr_r in enumerate(trs):
                    c_r, o_r, l_r = (tr_r[key].cpu().numpy() for key in ("counts", "offsets", "list"))
                    shift = r * n * k if g < E else r * n
                    got.extend((l_r[o_r[g]:o_r[g] + c_r[g]] + shift).tolist())
                assert np.array_equal(np.array(got, np.int64), want.astype(np.int64)), (t, l, g)
            st_full = full.get_state(l)
            for r, st in enumerate(ranks):
                st_r = st.get_state(l)
                for key in ("cache_e", "cache_w", "cache_norm", "cache_h", "ema"):
                    assert torch.equal(st_r[key], st_full[key][r * n:(r + 1) * n]), (t, l, r, key)
        reused += sum(st.stats()["reused"] for st in ranks) if t == 4 else 0
    assert reused > 0
    full.close()
    for st in ranks:
        st.close()


def test_shard_argument_checks(M):
    T, D, E, k, F = 128, 128, 8, 2, 128
    ws = [W.tiny_layer(610, T, D, E, k, F, dtype="bf16", wscale=0.05)[0]]
    st = _stack(M, ws, T, D, E, k, F, 0)
    nbytes = M.moeca_shard_exchange_bytes(st.handle, T)
    send = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    recv = torch.zeros(2 * nbytes, dtype=torch.uint8, device="cuda")
    x = torch.zeros((T, D), dtype=torch.bfloat16, device="cuda")
    out = torch.empty_like(x)
    with pytest.raises(M.MoecaError):  # rank out of range
        M.moeca_shard_begin(st.handle, x.data_ptr(), out.data_ptr(), T, 0, 2, 2, send.data_ptr(), recv.data_ptr())
    with pytest.raises(M.MoecaError):  # not a multiple of the token block
        M.moeca_shard_exchange_bytes(st.handle, T - 1)
    with pytest.raises(M.MoecaError):  # nothing begun
        M.moeca_shard_next(st.handle)
    st.close()
