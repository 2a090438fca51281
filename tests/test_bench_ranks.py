"""Multi-rank host logic of bench.py on CPU: two gloo ranks (replicas, no data-path collective).

Each rank scores its own events; the whole-job figures are the slowest rank's step time and the
units summed over ranks.  The GPU ranks use NCCL for the same two all-reduces.
"""
import importlib.util
import multiprocessing as mp
import os
import socket

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _load_bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench = _load_bench()
        # rank r: step of (r + 1) ms over (r + 1) * 1000 edges
        t, u = bench.whole_job((rank + 1) * 1e-3, (rank + 1) * 1000, world)
        dist.barrier()
        q.put((rank, t, u))
    finally:
        dist.destroy_process_group()


def test_whole_job_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=5) for _ in range(2))
    for rank, t, u in got:
        assert t == pytest.approx(2e-3)          # the slowest rank
        assert u == 3000                         # edges of both ranks
    # whole-job throughput = 3000 edges / 2 ms, not 2 x one rank's


def test_whole_job_single_rank_is_identity():
    bench = _load_bench()
    assert bench.whole_job(1.5e-3, 42, 1) == (1.5e-3, 42)
