"""The N > 1 path of bench.py on CPU: two gloo ranks, each with its own
shard of the job's assets (weak scaling over assets; no collective on the
data path), the job time is the maximum over ranks and the value counts
every rank's pixels.  Each rank runs the oracle on its shard, and the
shards together reproduce a single-process run of the whole batch."""
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
        assets = 2
    w = bench.workload(A, rank)
    # this rank's shard through the oracle (the first 6 steps of its trajectory)
    pixels, _, x, cache = bench.oracle_trajectory(w, steps=6, state=True)
    assets = list(range(w.first_asset, w.first_asset + w.B))
    q.put((rank, m, value, assets, pixels, x, cache))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_assets_and_take_the_max_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=300) for _ in procs), key=lambda r: r[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, m0, v0, a0, px0, x0, c0), (r1, m1, v1, a1, px1, x1, c1) = res
    assert m0 == m1 == 5.0                      # slowest rank
    assert v0 == v1 == pytest.approx(2 * 1000.0 / 5e-3)  # all ranks' pixels / job time
    # the shards partition the job's assets: disjoint, together 0 .. 3
    assert not set(a0) & set(a1) and sorted(a0 + a1) == [0, 1, 2, 3]
    # each shard's trajectory equals the single-process run of the whole
    # batch restricted to those assets (no asset processed twice or mixed up)
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_13255_gb300 import synth
    w_all = synth.make_workload("hunyuan64", B=4)
    px_all, _, x_all, c_all = bench.oracle_trajectory(w_all, steps=6, state=True)
    assert px0 + px1 == px_all > 0
    for assets, x, c in ((a0, x0, c0), (a1, x1, c1)):
        np.testing.assert_array_equal(x, x_all[assets])
        np.testing.assert_array_equal(c, c_all[assets])
