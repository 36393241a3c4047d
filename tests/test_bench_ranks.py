"""The multi-GPU bench path on the host: ranks split the sweep's traces, and
the whole-job figures are the slowest rank's time over the units of all ranks.
Run as two gloo ranks on the CPU (no GPU, no NCCL)."""
import os
import socket
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        # rank r: 10 + r ms, 100 + r records, 5 model-windows
        ms, units = bench.over_ranks(dist, "cpu", 10.0 + rank, [100 + rank, 5])
        ms_only, none = bench.over_ranks(dist, "cpu", 3.0 * (rank + 1), [])
        q.put((rank, ms, units, ms_only, none))
    finally:
        dist.destroy_process_group()


def test_over_ranks_two_gloo_ranks():
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
    for rank, ms, units, ms_only, none in out:
        assert ms == 11.0                     # the slowest rank's time
        assert units == [201.0, 10.0]         # every rank's units
        assert ms_only == 6.0 and none == []


def test_ranks_split_the_sweep_traces():
    """Every trace of the sweep goes to exactly one rank, for any rank count
    (ranks beyond the trace count get none and only join the collectives)."""
    sys.path.insert(0, ROOT)
    from paper_2609_29160_gb300 import partition
    for world in (1, 2, 4, 7, 8):
        got = sorted(t for r in range(world) for t in partition.sweep_traces(7, r, world))
        assert got == list(range(7))
        sizes = [len(partition.sweep_traces(7, r, world)) for r in range(world)]
        assert max(sizes) - min(sizes) <= 1


def _idle_worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    if rank == 1:
        bench.idle_rank(dist, world, "cpu")      # the idle rank's side, on the CPU
        q.put((rank, None, None))
        return
    dist.barrier()
    dist.barrier()
    ms, units = bench.over_ranks(dist, "cpu", 7.0, [10, 20, 30, 40, 50])
    e2e, _ = bench.over_ranks(dist, "cpu", 9.0, [])
    dist.destroy_process_group()
    q.put((rank, (ms, units), e2e))


def test_idle_rank_joins_the_collectives():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_idle_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = dict((r, (a, b)) for r, a, b in (q.get(timeout=120) for _ in procs))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (ms, units), e2e = out[0]
    assert ms == 7.0 and units == [10.0, 20.0, 30.0, 40.0, 50.0] and e2e == 9.0
