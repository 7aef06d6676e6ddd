"""The N > 1 path of the timing script on CPU: two gloo ranks, each a replica.

Every (slot, layer, head) update is independent, so ranks run replicas with no
collective on the data path; the only cross-rank step is the timing reduction
(max of the timed region over ranks) and the whole-job rate.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, times, results):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    total, value = bench.reduce_over_ranks(times[rank], 1000.0, world)
    results[rank] = (total, value)
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_timing_reduction_over_gloo_ranks(world):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        results = m.dict()
        times = [12.5, 20.0]
        port = _free_port()
        procs = [ctx.Process(target=_rank, args=(r, world, port, times, results)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
            assert p.exitcode == 0
        for r in range(world):
            total, value = results[r]
            assert total == 20.0                       # slowest rank's time on every rank
            assert abs(value - world * 1000.0 / 0.020) < 1e-6    # all ranks' units over it


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_over_ranks(10.0, 500.0, 1) == (10.0, 500.0 / 0.01)
