"""The bench's multi-GPU path is independent replicas (weak scaling, no
collective on the data path); its host logic -- max step time and summed units
over ranks -- runs here as world-size-2 gloo ranks on the CPU."""
import os
import socket

import pytest
import torch.distributed as dist
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
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, units = bench.aggregate(1.5 + rank, 18.0 * (rank + 1), world)
    q.put((rank, ms, units, bench.dist_env()))
    dist.destroy_process_group()


def test_aggregate_max_time_sum_units_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, ms, units, env in out:
        assert ms == pytest.approx(2.5)           # slowest rank
        assert units == pytest.approx(18.0 + 36.0)  # all ranks' positions
        assert env == (2, rank, rank)


def test_single_rank_aggregate_is_identity():
    import bench
    assert bench.aggregate(3.0, 7.0, 1) == (3.0, 7.0)
