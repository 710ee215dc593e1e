"""The N > 1 path of bench.py on CPU: two gloo ranks on 127.0.0.1.

The path shards as independent replicas (every rank simulates its own envs under its own
seed, with no data-path collective): each rank's result equals a single-process run of
its replica, the replicas differ from one another, every rank is charged the slowest
rank's time (max over ranks), and the job's value is all ranks' units over that time.
The oracle stands in for each rank's GPU work.
"""
import hashlib
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest

torch = pytest.importorskip("torch")

E, H = 6, 30


def _digest(out):
    h = hashlib.sha256()
    for k in ("action", "reward", "state"):
        h.update(np.ascontiguousarray(out[k]).tobytes())
    return h.hexdigest()


def _replica(seed):
    import oracle
    from paper_2607_05272_gb300 import workloads as W
    return oracle.rollout(W.c2(E), None, seed, 2, list(range(E)), H)   # Static baseline


def _worker(rank, world, port, q):
    import torch.distributed as dist

    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out = _replica(bench.replica_seed(rank))
        ms = 10.0 + 5.0 * rank                 # this rank's step time
        mx = bench.max_over_ranks(ms, dist)
        q.put((rank, _digest(out), mx, bench.job_value(world, E * H, mx)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_run_independent_replicas():
    import bench
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    ps = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in ps:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in ps:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[0] for r in res] == [0, 1]
    assert all(r[2] == 15.0 for r in res)                            # the slowest rank's time
    assert all(r[3] == world * E * H / 15e-3 for r in res)
    assert res[0][1] != res[1][1]                                     # independent replicas
    for rank, dig, _, _ in res:                                       # equal to a lone run
        assert dig == _digest(_replica(bench.replica_seed(rank)))


def test_single_rank_helpers():
    import bench
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.job_value(1, 2_097_152, 10.0) == pytest.approx(209_715_200.0)
    assert bench.replica_seed(3) - bench.replica_seed(0) == 3
