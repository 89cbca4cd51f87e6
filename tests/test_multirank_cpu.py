"""The bench's multi-rank aggregation over a world of 2 gloo ranks on CPU:
value = all ranks' positions / the slowest rank's time (no collective on the
data path; each rank decodes its own batch)."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, pos = bench.aggregate(10.0 + 5.0 * rank, 100 * (rank + 1), dist, "cpu")
    q.put((rank, ms, pos))
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_aggregation():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for _, ms, pos in out:
        assert ms == 15.0            # slowest rank
        assert pos == 300            # 100 + 200


def test_single_rank_passthrough():
    import bench
    assert bench.aggregate(3.5, 42) == (3.5, 42)


def _rank_fail(rank, world, port, q):
    # Rank 1 fails on the host before the aggregation (an exception ends its
    # process); rank 0 must get an error from its next collective within the
    # process-group timeout instead of waiting for ever.
    import time
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), CAI_PG_TIMEOUT_S="10")
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=bench.pg_timeout())
    if rank == 1:
        raise RuntimeError("rank 1 fails between steps")
    t0 = time.perf_counter()
    try:
        bench.aggregate(10.0, 100, dist, "cpu")
        q.put(("no error", time.perf_counter() - t0))
    except Exception as e:  # noqa: BLE001 - any collective error is the signal
        q.put((type(e).__name__, time.perf_counter() - t0))


def test_failed_rank_is_detected_not_waited_for():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_fail, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    kind, waited = q.get(timeout=120)
    for p in procs:
        p.join(timeout=60)
    assert kind != "no error" and waited < 60.0, (kind, waited)
    assert procs[1].exitcode != 0 and procs[0].exitcode == 0
