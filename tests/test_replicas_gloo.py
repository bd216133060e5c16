"""Multi-rank bookkeeping of bench.py on CPU: two gloo ranks, each with its own
part of the pool, reduce their work and time the way the GPU job does (sum of
rows, max of step times), and their parts are distinct draws."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_36830_gb300 import replicas, workloads
    ws, r, local = replicas.rank_env()
    pool = workloads.make_pool("tiny", seed=replicas.replica_seed("tiny", r))
    rows = workloads.make_rows(pool)
    local_rows = int(rows.mask.sum())
    local_ms = 10.0 + 5.0 * r
    total_rows, max_ms = replicas.job_totals(local_rows, local_ms)
    q.put((r, ws, local_rows, total_rows, max_ms, pool.c_version.tolist()))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_reduce_like_the_job():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    out.sort()
    assert all(o[1] == world for o in out)
    assert out[0][3] == out[1][3] == out[0][2] + out[1][2]  # rows summed over ranks
    assert out[0][4] == out[1][4] == 15.0                  # slowest rank's time
    assert out[0][5] != out[1][5]                          # independent pools


def test_single_process_totals_are_identity():
    from paper_2609_36830_gb300 import replicas
    assert replicas.job_totals(123, 4.5) == (123, 4.5)
    assert replicas.replica_seed("math7b", 0) == 20260001
    assert len({replicas.replica_seed("math7b", r) for r in range(8)}) == 8
