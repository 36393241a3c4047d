"""Property-based pins for the oracle (hypothesis explores small edge cases:
records on window boundaries, zero-length spans, one output token, spans past
the end of the grid, empty inputs). Each property ties the oracle to a
formulation other than its own: per-millisecond membership for the gauges and
the time-averaged occupancy, the closed-form decode staircase, conservation of
tokens, and the key-enumeration brute-force controller walk.
"""
import numpy as np
import pytest

hyp = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402

import oracle  # noqa: E402
from tests.test_oracle_reduce import _staircase_D  # noqa: E402
from tests.test_oracle_select import _brute_walk  # noqa: E402


@st.composite
def grids_and_records(draw, max_n=12):
    M = draw(st.integers(1, 3))
    win = draw(st.sampled_from([1, 3, 7, 10]))
    K = draw(st.integers(1, 12))
    span = K * win
    n = draw(st.integers(0, max_n))
    cols = {k: [] for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms",
                            "L_in", "L_out")}
    for _ in range(n):
        ta = draw(st.integers(0, span - 1))
        ts = ta + draw(st.integers(0, 2 * win + 1))
        tf = ts + draw(st.integers(0, 2 * win + 1))
        L = draw(st.integers(1, 9))
        te = tf if L == 1 else tf + draw(st.integers(0, 3 * win + 2))
        cols["model"].append(draw(st.integers(0, M - 1)))
        cols["t_arr_ms"].append(ta)
        cols["t_start_ms"].append(ts)
        cols["t_first_ms"].append(tf)
        cols["t_end_ms"].append(te)
        cols["L_in"].append(draw(st.integers(0, 20)))
        cols["L_out"].append(L)
    return M, win, K, {k: np.array(v, np.int32) for k, v in cols.items()}


def _membership(req, M, win, K):
    """Per-millisecond counts of running and waiting requests."""
    span = K * win
    run = np.zeros((span, M), np.int64)
    wait = np.zeros((span, M), np.int64)
    for i in range(len(req["model"])):
        m = req["model"][i]
        ta, ts, te = (int(req[k][i]) for k in ("t_arr_ms", "t_start_ms", "t_end_ms"))
        run[ts:min(te, span), m] += 1
        wait[ta:min(ts, span), m] += 1
    return run, wait


@settings(max_examples=120, deadline=None)
@given(grids_and_records())
def test_reduce_against_millisecond_membership_and_staircase(case):
    M, win, K, req = case
    P, D, A, W, drops = oracle.reduce_requests(req, M, win, K)
    assert drops.sum() == 0
    run, wait = _membership(req, M, win, K)
    last = np.arange(K) * win + win - 1                 # each window's last millisecond
    np.testing.assert_array_equal(A, run[last])
    np.testing.assert_array_equal(W, wait[last])
    np.testing.assert_array_equal(D, _staircase_D(req, M, win, K))
    span = K * win
    for m in range(M):
        sel = (req["model"] == m) & (req["t_first_ms"] < span)
        assert P[:, m].sum() == req["L_in"][sel].sum()


@settings(max_examples=120, deadline=None)
@given(grids_and_records())
def test_time_averaged_occupancy_against_millisecond_membership(case):
    M, win, K, req = case
    A_ms, W_ms = oracle.occupancy_mean_requests(req, M, win, K)
    run, wait = _membership(req, M, win, K)
    np.testing.assert_array_equal(A_ms, run.reshape(K, win, M).sum(axis=1))
    np.testing.assert_array_equal(W_ms, wait.reshape(K, win, M).sum(axis=1))


@st.composite
def walks(draw):
    M = draw(st.integers(1, 4))
    K = draw(st.integers(1, 40))
    win = draw(st.sampled_from([1000, 2500, 5000, 7000]))
    vals = [0.3, 0.5, 0.8, 0.9, 1.0, 1.1, 1.3, 2.0]
    Z = np.array([[draw(st.sampled_from(vals)) for _ in range(M)] for _ in range(K)])
    cls = np.array([[draw(st.sampled_from([1, 1, 1, 3])) for _ in range(M)] for _ in range(K)],
                   np.uint8)
    r0 = [draw(st.integers(0, 3)) for _ in range(M)]
    r_min = [draw(st.integers(0, 1)) for _ in range(M)]
    budget = sum(r0) + draw(st.integers(0, 2))
    Kp = draw(st.integers(0, 3))
    return Z, cls, win, budget, r0, r_min, Kp


@settings(max_examples=150, deadline=None)
@given(walks())
def test_walk_against_key_enumeration(w):
    Z, cls, win, budget, r0, r_min, Kp = w
    M = Z.shape[1]
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, budget, r0, r_min, np.ones(M),
                                    pacing_cap=Kp)
    want, r_want = _brute_walk(Z, cls, 0.8, 1.2, win, budget, r0, r_min, 5000, 10000, Kp)
    got = [(int(x["window"]), int(x["recv"]), int(x["donor"]), int(x["kind"]), int(x["seq"]))
           for x in mv]
    assert got == want
    assert rf.tolist() == r_want


@st.composite
def calibration_cases(draw):
    K = draw(st.integers(0, 25))
    M = draw(st.integers(1, 3))
    levels = [0.0, 0.25, 0.5, 1.0, 1.5, 2.0, 3.0]
    S = np.array([[draw(st.sampled_from(levels)) for _ in range(M)] for _ in range(K)],
                 np.float64).reshape(K, M)
    cls = np.array([[draw(st.sampled_from([1, 1, 3])) for _ in range(M)] for _ in range(K)],
                   np.uint8).reshape(K, M)
    n_arr = np.array([[draw(st.integers(0, 6)) for _ in range(M)] for _ in range(K)],
                     np.int32).reshape(K, M)
    n_met = np.array([[draw(st.integers(0, int(a))) for a in row] for row in n_arr],
                     np.int32).reshape(K, M)
    ok_frac = draw(st.sampled_from([0.5, 0.95, 1.0]))
    rho = draw(st.sampled_from([0.5, 0.8, 0.95, 1.0]))
    return S, cls, n_arr, n_met, ok_frac, rho


@settings(max_examples=200, deadline=None)
@given(calibration_cases())
def test_theta_against_brute_force(case):
    from tests.test_oracle_calibrate import _brute_theta
    S, cls, n_arr, n_met, ok_frac, rho = case
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, ok_frac, rho)
    want, wdeg = _brute_theta(S, cls, n_arr, n_met, ok_frac, rho)
    np.testing.assert_array_equal(theta, want)
    assert deg == wdeg


@st.composite
def latent_cases(draw):
    M = draw(st.integers(1, 3))
    K = draw(st.integers(1, 12))
    n = draw(st.integers(0, 10))
    rows = []
    for _ in range(n):
        d_total = draw(st.integers(0, 9000))
        rows.append((draw(st.integers(0, M - 1)), draw(st.integers(0, K * 1000 - 1)),
                     draw(st.integers(0, d_total)), d_total, draw(st.integers(0, 30)),
                     draw(st.integers(1, 6))))
    rows.sort(key=lambda r: r[1])
    cols = list(zip(*rows)) if rows else [[]] * 6
    lat = {k: np.array(v, np.int32) for k, v in zip(
        ("model", "t_arr_ms", "d_first_ms", "d_total_ms", "L_in", "L_out"), cols)}
    r0 = [draw(st.integers(0, 2)) for _ in range(M)]
    budget = sum(r0) + draw(st.integers(0, 1))
    Kp = draw(st.integers(0, 2))
    wake = draw(st.sampled_from([0, 700]))
    sleep = draw(st.sampled_from([0, 1200]))
    theta = draw(st.sampled_from([0.5, 5.0, 50.0]))
    return M, K, lat, r0, budget, Kp, wake, sleep, theta


@settings(max_examples=60, deadline=None)
@given(latent_cases())
def test_closed_loop_against_batch_rescoring(case):
    # decisions use only telemetry complete at their tick, with any delays
    M, K, lat, r0, budget, Kp, wake, sleep, theta = case
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.5, "theta": np.full(M, theta)}
    o = oracle.closed_loop(lat, M, 1000, K, prof, budget, r0, np.zeros(M, np.int32),
                           np.ones(M, np.int32), 0.8, 1.2, pacing_cap=Kp, wake_ms=wake,
                           sleep_ms=sleep)
    P, D, A, W, drops = oracle.reduce_requests(o["records"], M, 1000, K)
    assert drops.sum() == 0
    _, Z, cls, _ = oracle.score(P, D, A, W, dict(prof, tau_crit=0.8, tau_surplus=1.2), 1000,
                                np.float64)
    np.testing.assert_array_equal(Z, o["Z"])
    np.testing.assert_array_equal(cls, o["cls"])
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, budget, r0, np.zeros(M),
                                    np.ones(M), pacing_cap=Kp)
    np.testing.assert_array_equal(mv, o["moves"])
    np.testing.assert_array_equal(rf, o["r_final"])
