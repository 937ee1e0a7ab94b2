"""The N > 1 path of bench.py on CPU: two gloo ranks, each with its own
independent assets (weak scaling over assets; no collective on the data
path), the job time is the maximum over ranks and the value counts every
rank's pixels."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    assert bench.dist_env()[:2] == (rank, world)
    ms = [3.0, 5.0][rank]
    m = bench.reduce_max(ms, world)
    value = bench.job_value(1000.0, world, m / 1e3)

    class A:
        workload = "hunyuan64"
        assets = 1
    w = bench.workload(A, rank)
    q.put((rank, m, value, w.seed, float(np.abs(w.pos).sum())))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_assets_and_take_the_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, m0, v0, s0, h0), (r1, m1, v1, s1, h1) = res
    assert m0 == m1 == 5.0                      # slowest rank
    assert v0 == v1 == pytest.approx(2 * 1000.0 / 5e-3)  # all ranks' pixels / job time
    assert s0 != s1 and h0 != h1                # independent assets per rank
