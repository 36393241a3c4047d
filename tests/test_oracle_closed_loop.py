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
* guards and transfers in progress: a per-millisecond re-implementation of
  the controller (latency-guard breaches pre-empting rescue, lost-capacity
  rescue, donors held by their guard, rescues deferred while a rebalance
  transfer is in progress) makes the same moves and starts every request at
  the same millisecond, with each of those events exercised;
* hand-derived cases.
"""
import numpy as np
import pytest

import oracle
import tracegen

CRIT, NOM, SURP, IDLE = oracle.CRIT, oracle.NOM, oracle.SURP, oracle.IDLE
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
    np.testing.assert_array_equal(cls, o["cls"])
    # the delays hold capacity back: the served queue is not the immediate one
    o0 = oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, 3.0)), 64, lat["r0"],
                            np.ones(M, np.int32), np.ones(M, np.int32), 0.8, 1.2, pacing_cap=2)
    assert not np.array_equal(o0["records"]["t_start_ms"], o["records"]["t_start_ms"])


def _sim_closed_loop(lat, K, r0, r_min, budget, Z, cls, cap, wake, sleep, guard, tc=0.8,
                     ts=1.2):
    """The controller written out again, stepping through every millisecond
    (unit footprints), from the Z and regions the replay reports (pinned
    separately by re-scoring the served records):
      * rescue at a fast tick: a model whose first tokens in the window came
        later than its guard bound after arrival pre-empts everything (lowest Z
        among them); otherwise the lowest Z among critical models and models
        with requests waiting and no routable replica; while a rebalance
        transfer is in progress (its receiver's new server not yet serving) a
        rescue without a guard breach is deferred, and the slow loop still
        stays out of the tick;
      * rebalance at a slow tick without a rescue receiver: argmin Z over
        non-idle models if below 1;
      * sources: the idle pool, then idle, surplus and nominal donors as in
        the open-loop walk, never a donor whose guard is breached.
    Returns the moves, start times and counts of each kind of event."""
    span = K * WIN
    n = len(lat["model"])
    free_at = [[0] * int(r0[m]) for m in range(M)]
    queues = [list(np.flatnonzero(lat["model"] == m)) for m in range(M)]
    start = np.full(n, span, np.int64)
    late = np.zeros((K, M), np.int64)
    arrived = np.zeros(M, np.int64)
    started = np.zeros(M, np.int64)
    r = [int(x) for x in r0]
    pool = budget - sum(r)
    reb_until = 0
    moves, ev = [], {"hard": 0, "held": 0, "deferred": 0, "lost": 0}
    arr_sorted = sorted(range(n), key=lambda i: int(lat["t_arr_ms"][i]))
    ai = 0
    for t in range(span + 1):
        if t > 0 and t % WIN == 0:                  # window k = t/WIN - 1 ends here
            k = t // WIN - 1
            fast, slow = _ticks(k)
            if fast or slow:
                z, c = Z[k], cls[k]
                reg = [IDLE if c[m] == IDLE else CRIT if z[m] < tc else SURP if z[m] > ts
                       else NOM for m in range(M)]
                g = [guard is not None and late[k, m] > 0 for m in range(M)]
                lost = [r[m] == 0 and arrived[m] - started[m] > 0 for m in range(M)]
                mode, recv, hard = 0, None, False
                if fast:
                    cand = [(z[m], m) for m in range(M) if g[m]]
                    if cand:
                        hard = True
                    else:
                        cand = [(z[m], m) for m in range(M) if reg[m] == CRIT or lost[m]]
                    if cand:
                        recv = min(cand)[1]
                        if t < reb_until and not hard:
                            ev["deferred"] += 1
                        else:
                            mode = 1
                            ev["hard"] += hard
                            ev["lost"] += lost[recv] and reg[recv] != CRIT and not hard
                if mode == 0 and recv is None and slow:
                    cand = [(z[m], m) for m in range(M) if reg[m] != IDLE]
                    if cand and min(cand)[0] < 1:
                        mode, recv = 2, min(cand)[1]
                for seq in range(cap if mode else 0):
                    src = [((0,), -1)] if pool >= 1 else []
                    for d in range(M):
                        if d == recv or reg[d] == CRIT or r[d] <= r_min[d]:
                            continue
                        if g[d]:
                            ev["held"] += 1
                            continue
                        if reg[d] == IDLE:
                            src.append(((1, d), d))
                        elif reg[d] == SURP:
                            src.append(((2, -z[d], d), d))
                        elif mode == 1 or z[d] > z[recv]:
                            src.append(((3, -z[d], d), d))
                    if not src:
                        break
                    _, d = min(src)
                    gpu = t
                    if d < 0:
                        pool -= 1
                    else:
                        r[d] -= 1
                        b = min(free_at[d])
                        free_at[d].remove(b)
                        gpu = max(b, t) + sleep
                    r[recv] += 1
                    free_at[recv].append(gpu + wake)
                    if mode == 2:
                        reb_until = max(reb_until, gpu + wake)
                    moves.append((k, recv, d, mode, seq))
        if t == span:
            break
        while ai < n and lat["t_arr_ms"][arr_sorted[ai]] <= t:
            arrived[int(lat["model"][arr_sorted[ai]])] += 1
            ai += 1
        for m in range(M):
            q = queues[m]
            while q and lat["t_arr_ms"][q[0]] <= t:
                free = [j for j, b in enumerate(free_at[m]) if b <= t]
                if not free:
                    break
                i = q.pop(0)
                start[i] = t
                started[m] += 1
                free_at[m][free[0]] = t + int(lat["d_total_ms"][i])
                tf = t + int(lat["d_first_ms"][i])
                if guard is not None and tf < span and tf - int(lat["t_arr_ms"][i]) > guard[m]:
                    late[tf // WIN, m] += 1
    return moves, start, ev


def _ticks(k):
    return ((k + 1) * WIN) // 5000 > (k * WIN) // 5000, ((k + 1) * WIN) // 10000 > (k * WIN) // 10000


@pytest.mark.parametrize("wake,sleep,guard,seed", [(1310, 1870, None, 9), (1310, 1870, 2500, 9),
                                                   (0, 0, 1500, 10), (3000, 500, 4000, 11),
                                                   (4000, 3000, None, 9), (4000, 3000, 20000, 12)])
def test_guarded_controller_matches_a_per_millisecond_simulation(wake, sleep, guard, seed):
    lat, K = _latent(0.003, seed, 300.0)
    r_min = np.array([1, 0, 1, 0, 1, 0, 1, 0], np.int32)
    gms = None if guard is None else np.full(M, guard, np.int32)
    o = oracle.closed_loop(lat, M, WIN, K, _prof(np.full(M, 3.0)), 64, lat["r0"], r_min,
                           np.ones(M, np.int32), 0.8, 1.2, pacing_cap=2, wake_ms=wake,
                           sleep_ms=sleep, guard_ms=gms)
    # the signal the controller acted on is the batch score of the served records
    P, D, A, W, _ = oracle.reduce_requests(o["records"], M, WIN, K)
    prof = dict(_prof(np.full(M, 3.0)), tau_crit=0.8, tau_surplus=1.2)
    _, Z, cls, _ = oracle.score(P, D, A, W, prof, WIN, np.float64)
    np.testing.assert_array_equal(Z, o["Z"])
    moves, start, ev = _sim_closed_loop(lat, K, lat["r0"], r_min, 64, Z, cls, 2, wake, sleep,
                                        gms)
    got = [tuple(int(x) for x in mv) for mv in o["moves"]]
    assert got == moves
    np.testing.assert_array_equal(o["records"]["t_start_ms"], start)
    assert len(moves) > 10
    if guard is not None:
        assert ev["hard"] > 0 and ev["held"] > 0, ev
    if wake + sleep >= 7000 and guard is None:    # transfers outlast the 5 s rescue cadence
        assert ev["deferred"] > 0, ev


def test_hard_guard_preempts_a_critical_rescue_hand_case():
    """Two models, 1 s windows, one replica each and one in the pool, guard
    2 s. Window 4 (the fast tick at 5 s): model 0 runs a request but emits no
    token (raw 0, so Z = 0: critical); model 1 is surplus (Z = 6) but its
    request arriving at 2 s got its first token at 4.5 s, 2.5 s after arrival.
    Without a guard the pool goes to the critical model 0; with the guard the
    breach pre-empts it and the pool goes to model 1."""
    lat = {"model": np.array([1, 1, 0], np.int32), "t_arr_ms": np.array([0, 2000, 100], np.int32),
           "d_first_ms": np.array([100, 2500, 10], np.int32),
           "d_total_ms": np.array([1500, 3000, 6000], np.int32),
           "L_in": np.array([10, 10, 1], np.int32), "L_out": np.array([5, 5, 2], np.int32)}
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 1.0, "theta": np.array([1000.0, 1.0])}
    first = []
    for g in (None, [2000, 2000]):
        o = oracle.closed_loop(lat, 2, 1000, 10, prof, 3, [1, 1], [0, 0], [1, 1], 0.8, 1.2,
                               pacing_cap=1, guard_ms=g)
        assert o["Z"][4].tolist() == [0.0, 6.0] and o["cls"][4].tolist() == [CRIT, SURP]
        first.append(tuple(int(x) for x in o["moves"][0]))
    assert first == [(4, 0, -1, 1, 0), (4, 1, -1, 1, 0)]
