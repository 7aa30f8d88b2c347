"""Token-sharded exchange on CPU: two gloo ranks (world size 2).

Each rank takes its block-aligned half of a batch, forms the per-block
entropy partials (S_e, U_e) of Eq. 11 from its tokens' EMA statistic in
float32 with the same in-block order as the preparation kernel, exchanges
them with the binding's torch.distributed all-gather, and reduces every
rank's partials in global block order.  The sums must equal a single rank's
reduction over the whole batch bit for bit, the thresholds the oracle's
Eq. 11-12 on the whole batch, and each rank's decisions the whole batch's.
"""
import math
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")

TB = 32  # tokens per block of the preparation kernel


def block_partials(C_tok: np.ndarray, E: int) -> np.ndarray:
    """[blocks, E, 2] float32: per block, S and U summed as the kernel does
    (J = 128 / E interleaved runs over the block's tokens, added in run
    order)."""
    T = C_tok.shape[0]
    J = 128 // E
    out = np.zeros((T // TB, E, 2), np.float32)
    for b in range(T // TB):
        c = C_tok[b * TB:(b + 1) * TB].astype(np.float32)
        u = np.where(c > 0, c * np.log(np.where(c > 0, c, 1)).astype(np.float32), 0).astype(np.float32)
        for e in range(E):
            S = np.float32(0)
            U = np.float32(0)
            for j in range(J):
                s_j, u_j = np.float32(0), np.float32(0)
                for q in range(j, TB, J):
                    s_j = np.float32(s_j + c[q, e])
                    u_j = np.float32(u_j + u[q, e])
                S, U = np.float32(S + s_j), np.float32(U + u_j)
            out[b, e] = (S, U)
    return out


def reduce_global(part: np.ndarray) -> np.ndarray:
    """Every block's partials in global block order: J interleaved runs over
    blocks, added in run order (the kernel's order), [E, 2] float32."""
    nb, E, _ = part.shape
    J = 128 // E
    out = np.zeros((E, 2), np.float32)
    for e in range(E):
        for k2 in range(2):
            tot = np.float32(0)
            for j in range(J):
                run = np.float32(0)
                for b in range(j, nb, J):
                    run = np.float32(run + part[b, e, k2])
                tot = np.float32(tot + run)
            out[e, k2] = tot
    return out


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    from oracle import moeca_oracle as O
    from paper_2606_15615_gb300 import moeca as M
    from paper_2606_15615_gb300.workloads import tiny_layer
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        T, D, E, k = 256, 32, 8, 2
        w, x0, rng = tiny_layer(77, T, D, E, k, 16, wscale=0.4)
        prm = O.Params(top_k=k, tau0=0.62)
        # Two steps on the whole batch, with the oracle: the statistic C and the cache.
        st = O.Stack([w], prm, D, E)
        x1 = (x0 + 0.3 * rng.standard_normal(x0.shape)).astype(np.float32)
        st.step(x0, 0)
        pre = st.states[0].copy()
        _, infos = st.step(x1, 1)
        C = st.states[0].C.T  # [T, E]
        n = T // world
        mine = slice(rank * n, (rank + 1) * n)
        send = torch.from_numpy(block_partials(C[mine], E).reshape(-1).view(np.uint8).copy())
        recv = torch.zeros(world * send.numel(), dtype=torch.uint8)
        M.torch_allgather()(send, recv)
        gathered = recv.numpy().view(np.float32).reshape(-1, E, 2)
        sums = reduce_global(gathered)
        whole = reduce_global(block_partials(C, E))
        S, U = sums[:, 0].astype(np.float64), sums[:, 1].astype(np.float64)
        H = np.where(S > 0, np.log(np.where(S > 0, S, 1)) - U / np.where(S > 0, S, 1), 0)
        tau = prm.tau0 * (1 + prm.alpha * (2 * np.clip(H / math.log(T), 0, 1) - 1))
        # This rank's decisions with the exchanged thresholds.
        e_cur, w_cur = infos[0]["e"][mine], infos[0]["w"][mine]
        sel = O.select_branches(e_cur, w_cur, pre.cache_e[mine], pre.cache_w[mine], pre.cache_norm[mine], tau,
                                prm.lambda1, prm.lambda2, False)
        q.put((rank, sums.tobytes() == whole.tobytes(), float(np.abs(tau / infos[0]["tau"] - 1).max()),
               bool(np.array_equal(sel["recompute"], infos[0]["recompute"][mine])), int(gathered.shape[0])))
    finally:
        dist.destroy_process_group()


def test_two_rank_exchange_matches_single_rank():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, bit_exact, tau_err, same_decisions, n_blocks in sorted(res):
        assert bit_exact, f"rank {rank}: gathered sums differ from the single-rank reduction"
        assert tau_err < 1e-5, f"rank {rank}: tau off by {tau_err:.2e} relative"
        assert same_decisions, f"rank {rank}: decisions differ"
        assert n_blocks == 256 // TB
