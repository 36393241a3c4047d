"""The multi-GPU bench path on the host: ranks sweep disjoint traces, and the
whole-job figures are the slowest rank's time over the units of all ranks.
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


def test_rank_workloads_are_disjoint():
    sys.path.insert(0, ROOT)
    import bench
    import tracegen
    s0, s1 = bench.rank_seed0(0), bench.rank_seed0(1)
    assert not set(range(s0, s0 + 7)) & set(range(s1, s1 + 7))
    a = tracegen.sweep_workload(scale=0.002, n_traces=2, seed0=s0)
    b = tracegen.sweep_workload(scale=0.002, n_traces=2, seed0=s1)
    assert not np.array_equal(a["traces"][0]["t_arr_ms"], b["traces"][0]["t_arr_ms"])
