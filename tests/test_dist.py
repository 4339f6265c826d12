"""Multi-rank host logic on CPU (gloo, world size 2): requests shard across
ranks with no collective on the data path, and the benchmark's job time is the
slowest rank's."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import oracle.fe_oracle as O
from paper_2603_02565_gb300 import workloads as wl


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _run(rank, world, port, fn, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        q.put((rank, fn(rank, world)))
    finally:
        dist.destroy_process_group()


def spawn(fn, world=2):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_run, args=(r, world, port, fn, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return out


def _timing(rank, world):
    # rank 1 is the slow one; both must report the same whole-job value
    return bench.weak_scaling_value(100.0 if rank == 0 else 250.0, world, B=256, steps=10, dist=dist)


def test_job_time_is_the_slowest_rank():
    out = spawn(_timing)
    for rank in (0, 1):
        value, total_ms = out[rank]
        assert total_ms == 250.0
        assert value == pytest.approx(2 * 256 * 10 / 0.25)


def _shard_scores(rank, world):
    # each rank scores its half of the requests; gathering gives the full batch
    w = wl.make_workload("tiny", B=4)
    B = w.shape[0]
    mine = list(range(rank * B // world, (rank + 1) * B // world))
    s = O.evaluate(w.context[mine], w.pool[mine], w.cand_idx[mine], w.weights, w.cfg)[0]
    parts = [None] * world
    dist.all_gather_object(parts, s)
    return np.concatenate(parts)


def test_request_sharding_equals_whole_batch():
    out = spawn(_shard_scores)
    w = wl.make_workload("tiny", B=4)
    whole = O.evaluate(w.context, w.pool, w.cand_idx, w.weights, w.cfg)[0]
    for rank in (0, 1):
        np.testing.assert_allclose(out[rank], whole, rtol=1e-12)


def test_ranks_rotate_distinct_batches():
    B = 256
    for copy in range(12):
        assert bench.rank_copy_shift(0, copy, B) != bench.rank_copy_shift(1, copy, B)
