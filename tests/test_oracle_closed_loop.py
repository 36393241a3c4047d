"""Pins for the oracle's closed-loop replay (the controller of Sec. IV-B/IV-C
acting on the capacity that serves the requests whose telemetry it scores).

* controller off (pacing cap 0): the served records equal the generator's own
  FCFS queue of the same latent requests (tracegen.fcfs_records, a separate
  heap implementation in another language);
* causality and consistency: reducing and scoring the served records with the
  separately pinned batch functions gives the Z and classes the replay acted
  on, bit for bit, and the batch walk over them gives the replay's moves and
  final replicas -- so every decision used only telemetry complete at its tick;
* the queue under changing capacity: a per-millisecond simulation (donor
  servers taken and receiver servers given at the tick times the moves give,
  with drain, sleep and wake delays) starts every request at the same
  millisecond; with delays the decisions stay consistent with the served
  records;
* a hand-derived two-request case.
"""
import numpy as np
import pytest

import oracle
import tracegen

M, WIN = 8, 1000


def _latent(scale, seed, duration_s):
    spec = tracegen.spec_mid(scale=scale, seed=seed, duration_s=duration_s)
    return tracegen.gen_latent(spec), int(round(duration_s * 1000)) // WIN


def _prof(theta):
    return {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": np.asarray(theta, np.float64)}


def _run(lat, K, cap, dtype=np.float64, theta=3.0, budget=64, r_min=None):
    r_min = np.ones(M, np.int32) if r_min is None else r_min
    return oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, theta)), budget, lat["r0"], r_min,
                              np.ones(M, np.int32), 0.8, 1.2, pacing_cap=cap, dtype=dtype)


@pytest.mark.parametrize("seed", [5, 6])
def test_controller_off_is_the_open_loop_queue(seed):
    lat, K = _latent(0.01, seed, 600.0)
    o = _run(lat, K, 0)
    assert len(o["moves"]) == 0
    ref = tracegen.fcfs_records(lat, M, lat["r0"])
    got = o["records"]
    started = got["t_start_ms"] < K * WIN
    for k in ("t_start_ms", "t_first_ms", "t_end_ms"):
        np.testing.assert_array_equal(got[k][started], ref[k][started])
    assert (ref["t_start_ms"][~started] >= K * WIN).all()
    assert started.mean() > 0.8


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
@pytest.mark.parametrize("cap", [1, 3])
def test_decisions_use_only_complete_telemetry(dtype, cap):
    lat, K = _latent(0.01, 7, 900.0)
    o = _run(lat, K, cap, dtype)
    assert len(o["moves"]) > 10
    rec = o["records"]
    P, D, A, W, drops = oracle.reduce_requests(rec, M, WIN, K)
    assert drops.sum() == 0
    prof = dict(_prof(np.full(M, 3.0)), tau_crit=0.8, tau_surplus=1.2)
    _, Z, cls, _ = oracle.score(P, D, A, W, prof, WIN, dtype)
    np.testing.assert_array_equal(Z, o["Z"])
    np.testing.assert_array_equal(cls, o["cls"])
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, WIN, 64, lat["r0"], np.ones(M),
                                    np.ones(M), pacing_cap=cap)
    np.testing.assert_array_equal(rf, o["r_final"])
    np.testing.assert_array_equal(mv, o["moves"])


def _per_ms_queue(lat, K, r0, moves, wake=0, sleep=0):
    """Start times by stepping through every millisecond. At a tick time each
    transition first takes its released donor replicas (each the donor's
    server that frees first; its GPU returns `sleep` ms after it drains), then
    gives the receiver a server that frees `wake` ms after the GPU it needs is
    free (at the tick when the idle pool paid for it). Then queued requests
    take free servers."""
    span = K * WIN
    trans = {}                                   # (window, seq) -> [recv, donors]
    for mv in moves:
        key = (int(mv["window"]), int(mv["seq"]))
        t = trans.setdefault(key, [int(mv["recv"]), []])
        if int(mv["donor"]) >= 0:
            t[1].append(int(mv["donor"]))
    at = {}
    for (w, sq) in sorted(trans):
        at.setdefault((w + 1) * WIN, []).append(trans[(w, sq)])
    busy = [[0] * int(r0[m]) for m in range(M)]
    queues = [list(np.flatnonzero(lat["model"] == m)) for m in range(M)]
    start = np.full(len(lat["model"]), span, np.int64)
    for t in range(span):
        for recv, donors in at.get(t, []):
            gpu = t
            for d in donors:
                b = min(busy[d])
                busy[d].remove(b)
                gpu = max(gpu, max(b, t) + sleep)
            busy[recv].append(gpu + wake)
        for m in range(M):
            q = queues[m]
            while q and lat["t_arr_ms"][q[0]] <= t:
                free = [j for j, b in enumerate(busy[m]) if b <= t]
                if not free:
                    break
                i = q.pop(0)
                start[i] = t
                busy[m][free[0]] = t + int(lat["d_total_ms"][i])
    return start


@pytest.mark.parametrize("wake,sleep", [(0, 0), (1310, 1870), (40, 0)])
def test_queue_under_changing_capacity_matches_per_millisecond_stepping(wake, sleep):
    lat, K = _latent(0.002, 8, 240.0)
    o = oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, 3.0)), 64, lat["r0"],
                           np.ones(M, np.int32), np.ones(M, np.int32), 0.8, 1.2, pacing_cap=2,
                           wake_ms=wake, sleep_ms=sleep)
    assert len(o["moves"]) > 0
    got = o["records"]["t_start_ms"]
    want = _per_ms_queue(lat, K, lat["r0"], o["moves"], wake, sleep)
    np.testing.assert_array_equal(got, want)


def test_actuation_delays_keep_decisions_consistent_with_the_served_records():
    lat, K = _latent(0.01, 9, 900.0)
    o = oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, 3.0)), 64, lat["r0"],
                           np.ones(M, np.int32), np.ones(M, np.int32), 0.8, 1.2, pacing_cap=2,
                           wake_ms=1310, sleep_ms=1870)
    P, D, A, W, _ = oracle.reduce_requests(o["records"], M, WIN, K)
    prof = dict(_prof(np.full(M, 3.0)), tau_crit=0.8, tau_surplus=1.2)
    _, Z, cls, _ = oracle.score(P, D, A, W, prof, WIN, np.float64)
    np.testing.assert_array_equal(Z, o["Z"])
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, WIN, 64, lat["r0"], np.ones(M),
                                    np.ones(M), pacing_cap=2)
    np.testing.assert_array_equal(mv, o["moves"])
    # the delays hold capacity back: the served queue is not the immediate one
    o0 = oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, 3.0)), 64, lat["r0"],
                            np.ones(M, np.int32), np.ones(M, np.int32), 0.8, 1.2, pacing_cap=2)
    assert not np.array_equal(o0["records"]["t_start_ms"], o["records"]["t_start_ms"])


def test_hand_case():
    # one model, one replica, windows of 1 s: request 0 occupies the server
    # from 0 to 3000 ms, request 1 (arrives at 500) waits for it
    lat = {"model": np.array([0, 0], np.int32), "t_arr_ms": np.array([0, 500], np.int32),
           "d_first_ms": np.array([100, 50], np.int32),
           "d_total_ms": np.array([3000, 1000], np.int32),
           "L_in": np.array([10, 10], np.int32), "L_out": np.array([5, 5], np.int32)}
    o = oracle.closed_loop(lat, 1, 1000, 6, _prof([1.0]), 1, [1], [1], [1], 0.8, 1.2,
                           pacing_cap=1)
    r = o["records"]
    assert r["t_start_ms"].tolist() == [0, 3000]
    assert r["t_first_ms"].tolist() == [100, 3050]
    assert r["t_end_ms"].tolist() == [3000, 4000]
    assert len(o["moves"]) == 0            # a single model has no donor and no pool
