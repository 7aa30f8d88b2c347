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
