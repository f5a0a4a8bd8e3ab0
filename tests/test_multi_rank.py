"""The N > 1 bench path on CPU with gloo, world size 2: requests are
partitioned across ranks (each rank its own seeded workload, no data-path
collective); the job's time is the max over ranks; the value counts every
rank's sequences."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    from synthetic import request_spans
    dist.init_process_group("gloo")
    try:
        # every rank times its own replica; the job time is the slowest
        t = bench.max_over_ranks(10.0 + rank, world)
        bench.barrier(world)
        # each rank's workload seed differs, so replicas hold different data
        seed = 0 + 1000 * rank
        spans = request_spans(seed, 0, 131072, 64)
        q.put((rank, t, spans[:3]))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    assert res[0][1] == res[1][1] == 11.0
    assert res[0][2] != res[1][2]


def _worker_fail(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import datetime

    import bench
    dist.init_process_group("gloo", timeout=datetime.timedelta(seconds=5))
    if rank == 1:
        q.put((rank, "left"))
        q.close()
        q.join_thread()
        os._exit(0)                # leaves between steps, without a word
    try:
        bench.max_over_ranks(1.0, world)
        q.put((rank, "no error"))
    except Exception:               # the survivor's collective ends with an error
        q.put((rank, "error"))
    q.close()
    q.join_thread()
    os._exit(0)


def test_rank_that_leaves_is_detected_by_the_other():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker_fail, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    res = dict(q.get(timeout=10) for _ in range(2))
    assert res == {0: "error", 1: "left"}
