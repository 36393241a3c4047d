"""The multi-GPU partition on the host, as two and three gloo ranks on the CPU
(no GPU): a long 64-model token stream split by model blocks, each rank
computing its models' signal, the exchange of Z and region rows at control
ticks, and the walk over the gathered tick rows. The per-rank computation here
is the oracle (a CPU stand-in for the library, which the GPU test runs); the
result must equal the unsplit oracle path: every model's counts, theta, Z and
regions, and the controller's moves and final replicas."""
import os
import socket
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
FAST, SLOW = 5000, 10000


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _workload():
    import tracegen
    w = tracegen.workload("stream", scale=0.002)
    # a shorter grid keeps the oracle quick: the first 4 h of the day
    w["K"] = 144000
    return w


def _oracle_signal(ev, M, win, K, slo, prof):
    import oracle
    P, D, A, W, _ = oracle.reduce_events(ev, M, win, K)
    n_arr, n_met = oracle.slo_counts_events(ev, M, win, K, slo)
    S, _, cls, _ = oracle.score(P, D, A, W, prof, win, np.float32)
    theta, _ = oracle.calibrate(S, cls, n_arr, n_met)
    _, Z, cls, _ = oracle.score(P, D, A, W, dict(prof, theta=theta), win, np.float32)
    return {"P": P, "D": D, "A": A, "W": W, "theta": theta, "Z": Z, "cls": cls}


def _worker(rank, world, port, q):
    try:
        _work(rank, world, port, q)
    except Exception as e:        # report, so the parent does not wait for nothing
        q.put((rank, "error", repr(e)))
        raise


def _work(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        import tracegen
        from paper_2609_29160_gb300 import partition
        w = _workload()
        M, win, K = w["M"], w["window_ms"], w["K"]
        blocks = partition.model_blocks(M, world)
        m0, m1 = blocks[rank]
        ev = partition.events_for_models(w["events"], m0, m1)
        prof = tracegen.default_profile(m1 - m0, win)
        sig = _oracle_signal(ev, m1 - m0, win, K, w["slo_ttft_ms"][m0:m1], prof)
        ticks = partition.tick_windows(K, win, FAST, SLOW)
        Zt = torch.as_tensor(np.ascontiguousarray(sig["Z"][ticks]))
        ct = torch.as_tensor(np.ascontiguousarray(sig["cls"][ticks]))
        Z, cls = partition.gather_tick_rows(dist, Zt, ct, blocks)
        full = tracegen.default_profile(M, win)
        mv, rf, _ = oracle.select_moves(Z.numpy(), cls.numpy(), 0.8, 1.2, FAST, w["budget"],
                                        w["r0"], w["r_min"], w["footprint"], FAST, SLOW, 1)
        mv = partition.moves_to_windows(mv, win, FAST)
        q.put((rank, (m0, m1), {k: sig[k] for k in ("P", "D", "A", "W", "theta")},
               Z.numpy(), cls.numpy(), mv, rf, full["w_p"][0]))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_model_partition_matches_the_unsplit_path(world):
    sys.path.insert(0, ROOT)
    import oracle
    import tracegen
    from paper_2609_29160_gb300 import partition
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted([q.get(timeout=300) for _ in procs], key=lambda x: x[0])
    errors = [o for o in out if o[1] == "error"]
    assert not errors, errors
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    w = _workload()
    M, win, K = w["M"], w["window_ms"], w["K"]
    ref = _oracle_signal(w["events"], M, win, K, w["slo_ttft_ms"],
                         tracegen.default_profile(M, win))
    mv, rf, _ = oracle.select_moves(ref["Z"], ref["cls"], 0.8, 1.2, win, w["budget"], w["r0"],
                                    w["r_min"], w["footprint"], FAST, SLOW, 1)
    assert len(mv) > 0
    ticks = partition.tick_windows(K, win, FAST, SLOW)
    for rank, (m0, m1), sig, Z, cls, mvr, rfr, _ in out:
        for k in ("P", "D", "A", "W"):
            np.testing.assert_array_equal(sig[k], ref[k][:, m0:m1], err_msg=f"{rank} {k}")
        np.testing.assert_array_equal(sig["theta"], ref["theta"][m0:m1])
        # every rank holds the same gathered rows and makes the same moves
        np.testing.assert_array_equal(Z, ref["Z"][ticks])
        np.testing.assert_array_equal(cls, ref["cls"][ticks])
        np.testing.assert_array_equal(mvr, mv)
        np.testing.assert_array_equal(rfr, rf)


def test_blocks_and_slices_cover_every_model_and_event_once():
    sys.path.insert(0, ROOT)
    from paper_2609_29160_gb300 import partition
    for M, n in ((64, 8), (64, 3), (5, 8), (1, 1)):
        blocks = partition.model_blocks(M, n)
        assert blocks[0][0] == 0 and blocks[-1][1] == M
        assert all(b[1] == c[0] for b, c in zip(blocks, blocks[1:]))
        sizes = [m1 - m0 for m0, m1 in blocks]
        assert max(sizes) - min(sizes) <= 1
    w = _workload()
    ev = w["events"]
    blocks = partition.model_blocks(w["M"], 3)
    parts = [partition.events_for_models(ev, m0, m1) for m0, m1 in blocks]
    assert sum(len(p["model"]) for p in parts) == len(ev["model"])
    assert sum(len(p["req_model"]) for p in parts) == len(ev["req_model"])
    for (m0, m1), p in zip(blocks, parts):
        # local request ids point at local requests of the same model
        assert (p["req"] >= 0).all()
        np.testing.assert_array_equal(p["req_model"][p["req"]], p["model"])
    assert partition.sweep_traces(7, 0, 3) == [0, 3, 6]
    assert sorted(sum((partition.sweep_traces(7, r, 3) for r in range(3)), [])) == list(range(7))


def test_tick_series_walk_equals_the_full_walk():
    """The walk reads nothing but fast-tick windows: on a series of only those
    windows, with the fast cadence as its window length, it makes the same
    moves (mapped back to the original windows)."""
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2609_29160_gb300 import partition
    rng = np.random.default_rng(4)
    K, M, win = 20000, 12, 100
    Z = rng.choice(np.array([0.3, 0.6, 0.8, 0.95, 1.0, 1.1, 1.3, 2.0]), (K, M)).astype(np.float32)
    cls = np.where(rng.random((K, M)) < 0.1, oracle.IDLE, oracle.NOM).astype(np.uint8)
    r0 = rng.integers(1, 6, M).astype(np.int32)
    args = (int(r0.sum()) + 2, r0, np.ones(M, np.int32), np.ones(M, np.int32))
    for cap in (1, 3):
        mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, *args, FAST, SLOW, cap)
        t = partition.tick_windows(K, win, FAST, SLOW)
        mt, rt, _ = oracle.select_moves(np.ascontiguousarray(Z[t]), np.ascontiguousarray(cls[t]),
                                        0.8, 1.2, FAST, *args, FAST, SLOW, cap)
        np.testing.assert_array_equal(partition.moves_to_windows(mt, win, FAST), mv)
        np.testing.assert_array_equal(rt, rf)
