"""bench.py's multi-rank bookkeeping on CPU: two gloo ranks, max time, summed tokens."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    w, r, l = bench.dist_env()
    d = bench.init_group(w, "gloo")
    ms, tokens = bench.aggregate(10.0 + 5.0 * rank, 1000 * (rank + 1), d)
    q.put((r, ms, tokens))
    d.barrier()
    d.destroy_process_group()


def test_two_gloo_ranks_take_max_time_and_sum_tokens():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got == [(0, 15.0, 3000), (1, 15.0, 3000)]


def test_single_rank_needs_no_group():
    import bench
    assert bench.init_group(1, "gloo") is None
    assert bench.aggregate(3.5, 77, None) == (3.5, 77)


def test_ffn_algorithmic_bytes_exclude_the_hidden_activations():
    """The grouped FFN's algorithmic bytes are the active experts' weights,
    the gathered input rows and the scattered output rows; its bf16 hidden
    activations are an implementation intermediate (not counted)."""
    import bench
    from paper_2606_15615_gb300 import workloads as W
    wl = W.workload(2)
    rows, G = 1638.4, 16
    b, f = bench.algorithmic("ffn", wl, rows, G)
    D, F = wl.hidden, wl.ffn
    assert b == 2 * G * F * D * 2 + 2 * rows * D * 2
    assert f == 4.0 * rows * D * F
    # 16 experts x 2 x 3072 x 768 x 2 B = 151.0 MB of weights, plus 2 x 1638.4 rows x 768 x 2 B.
    assert abs(b / 1e6 - 156.03) < 0.05


def test_roofline_uses_burst_peaks_and_bounds():
    import bench
    from paper_2606_15615_gb300 import workloads as W
    pk = {"hbm_gbs": 6694.5, "bf16_tflops": 1918.9, "bf16_tflops_sustained": 1733.4}
    wl = W.workload(2)
    kd = {"alg_bytes": 156.0e6, "alg_flops": 15.46e9, "avg_us": 50.0, "gbs": 3120.0, "tflops": 309.2}
    r = bench.roofline("ffn", kd, wl, pk, "measured", None)
    assert r["bound"] == "hbm" and r["peak"] == 6694.5 and abs(r["frac"] - 3120.0 / 6694.5) < 1e-12
    kd4 = {"alg_bytes": 400e6, "alg_flops": 350e12 * 1e-3, "avg_us": 300.0, "gbs": 1333.0, "tflops": 1166.7}
    r4 = bench.roofline("ffn", kd4, W.workload(4), pk, "measured", None)
    assert r4["bound"] == "tensor" and r4["peak"] == 1918.9  # burst, not sustained
    kd1 = {"alg_bytes": 20e6, "alg_flops": 1.2e9, "avg_us": 60.0, "gbs": 333.0, "tflops": 20.0}
    r1 = bench.roofline("ffn2", kd1, W.workload(1), pk, "measured", 75.0)
    assert r1["bound"] == "fp32" and abs(r1["frac"] - 20.0 / 75.0) < 1e-12
