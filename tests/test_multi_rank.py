"""Host logic of bench.py under torch.distributed with N > 1, on CPU (gloo,
world size 2): every rank quantises its own copy of the workload (weak
scaling, no collective on the data path), the step time is the slowest rank's
and the reported value counts the elements of all ranks."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local_ms = 10.0 + 5.0 * rank            # rank 1 is slower
    dist.barrier()
    ms = bench.reduce_max_ms(local_ms, world, "cpu")
    elems = 1000
    value = world * elems / (ms * 1e-3) / 1e9
    q.put((rank, ms, value))
    dist.barrier()
    dist.destroy_process_group()


def test_weak_scaling_timing_is_max_over_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [15.0, 15.0]          # every rank sees the slowest rank's time
    assert res[0][2] == pytest.approx(2 * 1000 / 15e-3 / 1e9)


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max_ms(3.5, 1, "cpu") == 3.5
