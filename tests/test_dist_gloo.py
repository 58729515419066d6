"""Multi-process host logic of bench.py on CPU: two gloo ranks.

The path runs as independent replicas (one per GPU, no data-path collective);
what crosses ranks is the timing: a barrier around the timed region and the
maximum of the per-rank step times, from which the whole-job throughput is
computed.  The reference arm runs on rank 0 only.
"""
import json
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    ws, r = bench.init_dist("gloo")
    assert (ws, r) == (world, rank)
    bench.barrier()
    ms = 1.0 + rank                          # rank 1 is the slowest
    ms_max = bench.max_over_ranks(ms)
    total = bench.sum_over_ranks(10.0)
    value = bench.job_throughput(1000, ms_max, ws)
    q.put((rank, ms_max, total, value))
    dist.destroy_process_group()


def test_max_over_ranks_and_throughput():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms_max, total, value in out:
        assert ms_max == 2.0                 # every rank sees the slowest rank's time
        assert total == 20.0
        assert value == pytest.approx(1000 * 2 / 2e-3)   # all ranks' units over the slowest time


def _reference_worker(rank, world, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import argparse
    import bench
    args = argparse.Namespace(workload="c1", kappa=None, steps=3, warmup=3, dtype=None)
    res, r = bench.run_reference(args)
    q.put((r, json.dumps(res) if res else None))


def test_reference_arm_runs_on_rank0_only():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_reference_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=300) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert out[1] is None
    res = json.loads(out[0])
    assert res["impl"] == "reference" and res["value"] > 0 and res["n_gpus"] == 2
    assert res["cpu_baseline"]["kind"] == "oracle" and res["e2e"]["h2d_bytes_per_step"] == 0
