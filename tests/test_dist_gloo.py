"""Multi-process host logic of bench.py on CPU (gloo, world size 2): the
max/sum reductions and barrier used around the timed region, the whole-job
aggregation of the metric, and the replicas' independent query batches.  The
path shards into independent problems, so these are the only cross-rank
operations (no collective on the data path)."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
import workloads as W  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, local = bench.dist_env()
    # per-rank step time and roofline time (ms, seconds), as the bench has them
    ms = 10.0 + 5.0 * rank
    rt = 0.004 + 0.001 * rank
    bench.barrier(w)
    ms_max = bench.reduce_max(ms, w)
    rt_sum = bench.reduce_sum(rt, w)
    value = bench.aggregate_value(rt_sum, ms_max)
    bench.barrier(w)
    out.put((rank, w, r, local, ms_max, rt_sum, value))
    dist.destroy_process_group()


def test_reductions_and_aggregate_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, w, r, local, ms_max, rt_sum, value in res:
        assert (w, r, local) == (2, rank, rank)
        assert ms_max == 15.0                    # slowest rank sets the step time
        assert abs(rt_sum - 0.009) < 1e-15       # roofline time of both replicas
        # whole-job % of one GPU's roofline: 100 * 9 ms / 15 ms
        assert abs(value - 60.0) < 1e-9
    assert res[0][4:] == res[1][4:]              # every rank holds the same aggregate


def test_single_process_is_identity():
    assert bench.reduce_max(3.5, 1) == 3.5
    assert bench.reduce_sum(2.0, 1) == 2.0
    bench.barrier(1)
    assert bench.aggregate_value(0.005, 10.0) == pytest.approx(50.0)


def test_replica_batches_are_independent():
    cfg = W.MATRIX_CONFIGS["tiny"]
    x0 = W.queries(cfg)
    x0b = W.queries(cfg, replica=0)
    x1 = W.queries(cfg, replica=1)
    assert np.array_equal(x0, x0b)               # replica 0 is the configuration's batch
    assert x1.shape == x0.shape
    assert not np.allclose(x0, x1)
    # independent draws: no more correlation than chance
    c = np.corrcoef(x0.ravel(), x1.ravel())[0, 1]
    assert abs(c) < 0.05
