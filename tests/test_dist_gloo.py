"""The multi-GPU benchmark path's host logic on CPU: two ranks over gloo.
Requests are independent, so ranks share nothing but the timing reduction:
the job's time is the slowest rank's, positions add up across ranks, and each
rank's requests take disjoint Philox request indices."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    r, ws, local = bench.dist_env()
    bench.dist_init(ws, "gloo")
    bench.barrier(ws)
    t = bench.max_over_ranks(1.0 + rank, ws)
    s = bench.sum_over_ranks(10.0 * (rank + 1), ws)
    q.put((r, ws, t, s, bench.request_base(r, 64)))
    import torch.distributed as dist
    dist.destroy_process_group()


def test_two_ranks_over_gloo():
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
    assert [r[0] for r in res] == [0, 1]
    assert all(r[1] == 2 for r in res)
    assert all(r[2] == 2.0 for r in res)  # max over ranks
    assert all(r[3] == 30.0 for r in res)  # positions add up
    assert res[0][4] == 0 and res[1][4] == 64  # disjoint request indices


def test_single_process_needs_no_group():
    import bench
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.sum_over_ranks(2.0, 1) == 2.0
