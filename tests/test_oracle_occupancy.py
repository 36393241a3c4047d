"""Pins for the oracle's time-averaged occupancy (the window-mean reading of
the running and waiting counts of Eq. 1, Sec. III-A) and for scoring with it.

* brute force: count the running and waiting requests at every millisecond
  and sum them per window (a different formulation from the oracle's
  per-window overlaps);
* one-millisecond windows: the window mean is the count at the window's only
  millisecond, i.e. the sampled gauge of the (separately pinned) reduction,
  and scoring with it equals scoring with the sampled gauges bit for bit;
* totals: the sum over windows is the length of each span inside the grid;
* the hand-derived worked example (tests/golden/w1_mean_occupancy.json);
* skipped records: a record the reduction drops adds nothing here either.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests.conftest import GOLDEN

KEYS = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")


def _valid_requests(rng, n, M, win, K, reach=3):
    span = K * win
    ta = rng.integers(0, span, n)
    ts = ta + rng.integers(0, reach * win, n) * (rng.random(n) < 0.7)
    tf = ts + rng.integers(0, 2 * win, n)
    te = tf + rng.integers(0, reach * win, n)
    # some spans run past the end of the grid
    te = np.where(rng.random(n) < 0.1, te + span, te)
    return {"model": rng.integers(0, M, n).astype(np.int32), "t_arr_ms": ta.astype(np.int32),
            "t_start_ms": ts.astype(np.int32), "t_first_ms": tf.astype(np.int32),
            "t_end_ms": te.astype(np.int32),
            "L_in": rng.integers(0, 50, n).astype(np.int32),
            "L_out": rng.integers(1, 20, n).astype(np.int32)}


def _brute(req, M, win, K):
    span = K * win
    A = np.zeros((K, M), np.int64)
    W = np.zeros((K, M), np.int64)
    for t in range(span):
        k = t // win
        for i in range(len(req["model"])):
            m = req["model"][i]
            if req["t_start_ms"][i] <= t < req["t_end_ms"][i]:
                A[k, m] += 1
            if req["t_arr_ms"][i] <= t < req["t_start_ms"][i]:
                W[k, m] += 1
    return A, W


@pytest.mark.parametrize("seed,M,win,K", [(0, 1, 7, 9), (1, 3, 5, 12), (2, 2, 13, 6), (3, 4, 1, 40)])
def test_matches_per_millisecond_brute_force(seed, M, win, K):
    rng = np.random.default_rng(seed)
    req = _valid_requests(rng, 40, M, win, K)
    A_ms, W_ms = oracle.occupancy_mean_requests(req, M, win, K)
    bA, bW = _brute(req, M, win, K)
    np.testing.assert_array_equal(A_ms, bA)
    np.testing.assert_array_equal(W_ms, bW)


@pytest.mark.parametrize("seed", range(4))
def test_one_millisecond_windows_equal_the_sampled_gauges(seed):
    rng = np.random.default_rng(10 + seed)
    M, K = 3, 400
    req = _valid_requests(rng, 300, M, 1, K, reach=40)
    _, _, A, W, _ = oracle.reduce_requests(req, M, 1, K)
    A_ms, W_ms = oracle.occupancy_mean_requests(req, M, 1, K)
    np.testing.assert_array_equal(A_ms, A)
    np.testing.assert_array_equal(W_ms, W)


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_scoring_with_one_millisecond_means_equals_sampled_scoring(dtype):
    rng = np.random.default_rng(21)
    M, K = 4, 300
    req = _valid_requests(rng, 200, M, 1, K, reach=30)
    P, D, A, W, _ = oracle.reduce_requests(req, M, 1, K)
    occ = oracle.occupancy_mean_requests(req, M, 1, K)
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.3, "theta": 1.7, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    ref = oracle.score(P, D, A, W, prof, 1, dtype)
    got = oracle.score(P, D, A, W, prof, 1, dtype, occ_ms=occ)
    for a, b in zip(ref, got):
        np.testing.assert_array_equal(a, b)


def test_totals_are_the_span_lengths_inside_the_grid():
    rng = np.random.default_rng(5)
    M, win, K = 5, 100, 300
    req = _valid_requests(rng, 2000, M, win, K, reach=20)
    A_ms, W_ms = oracle.occupancy_mean_requests(req, M, win, K)
    span = K * win
    clip = lambda a, b: np.clip(np.minimum(b, span) - a, 0, None).astype(np.int64)
    run = clip(req["t_start_ms"].astype(np.int64), req["t_end_ms"].astype(np.int64))
    wait = clip(req["t_arr_ms"].astype(np.int64), req["t_start_ms"].astype(np.int64))
    for m in range(M):
        sel = req["model"] == m
        assert A_ms[:, m].sum() == run[sel].sum()
        assert W_ms[:, m].sum() == wait[sel].sum()
    assert (A_ms >= 0).all() and (W_ms >= 0).all()
    assert (A_ms <= 2000 * win).all()


def test_worked_example():
    with open(os.path.join(GOLDEN, "w1_worked_example.json")) as f:
        w1 = json.load(f)
    with open(os.path.join(GOLDEN, "w1_mean_occupancy.json")) as f:
        g = json.load(f)
    req = {k: np.array(v, np.int32) for k, v in w1["requests"].items()}
    e = g["expected"]
    A_ms, W_ms = oracle.occupancy_mean_requests(req, 1, 1000, 3)
    assert A_ms[:, 0].tolist() == e["A_ms"] and W_ms[:, 0].tolist() == e["W_ms"]
    P, D, A, W, _ = oracle.reduce_requests(req, 1, 1000, 3)
    for dtype, rtol in ((np.float64, 1e-14), (np.float32, 1e-6)):
        S, Z, cls, _ = oracle.score(P, D, A, W, g["profile"], 1000, dtype, occ_ms=(A_ms, W_ms))
        for k in range(3):
            s = Fraction(e["S_num"][k], e["S_den"][k])
            assert S[k, 0] == pytest.approx(float(s), rel=rtol)
            assert Z[k, 0] == pytest.approx(float(s / 20), rel=rtol)
        assert cls[:, 0].tolist() == e["cls"]


def test_dropped_records_add_nothing():
    rng = np.random.default_rng(8)
    M, win, K = 3, 50, 40
    good = _valid_requests(rng, 100, M, win, K)
    bad = _valid_requests(rng, 30, M, win, K)
    bad["model"][:10] = M + 1                      # bad model id
    bad["t_arr_ms"][10:20] = K * win + 5           # arrival past the grid
    bad["t_start_ms"][10:20] = K * win + 6
    bad["t_first_ms"][10:20] = K * win + 7
    bad["t_end_ms"][10:20] = K * win + 8
    bad["t_end_ms"][20:25] = bad["t_first_ms"][20:25] - 1   # order violation
    bad["L_out"][25:30] = 0                        # bad length
    both = {k: np.concatenate([good[k], bad[k]]) for k in KEYS}
    _, _, _, _, drops = oracle.reduce_requests(both, M, win, K)
    assert drops.sum() == 30
    np.testing.assert_array_equal(np.stack(oracle.occupancy_mean_requests(both, M, win, K)),
                                  np.stack(oracle.occupancy_mean_requests(good, M, win, K)))


def _events_case(seed, scale=0.002):
    import tracegen
    return tracegen.workload("stream", scale=scale, seed=seed)


def test_events_one_millisecond_windows_equal_the_sampled_gauges():
    # with 1 ms windows the window mean is the count at its only millisecond
    w = _events_case(5)
    ev, M = w["events"], w["M"]
    K = 20000                                   # the first 20 s, 1 ms windows
    _, _, A, W, _ = oracle.reduce_events(ev, M, 1, K)
    A_ms, W_ms = oracle.occupancy_mean_events(ev, M, 1, K)
    np.testing.assert_array_equal(A_ms, A)
    np.testing.assert_array_equal(W_ms, W)


def test_events_against_per_millisecond_membership():
    w = _events_case(6)
    ev, M = w["events"], w["M"]
    win, K = 250, 60
    span = win * K
    A_ms, W_ms = oracle.occupancy_mean_events(ev, M, win, K)
    # spans from the valid events of each request (numpy group min / max)
    t = np.floor(ev["t_s"].astype(np.float64) * 1000.0)
    ok = (t >= 0) & (t < span) & (ev["phase"] <= 1) & (ev["model"] == ev["req_model"][ev["req"]])
    n_req = len(ev["req_model"])
    first = np.full(n_req, np.iinfo(np.int64).max)
    last = np.full(n_req, -1)
    np.minimum.at(first, ev["req"][ok], t[ok].astype(np.int64))
    np.maximum.at(last, ev["req"][ok], t[ok].astype(np.int64))
    run = np.zeros((span, M), np.int64)
    wait = np.zeros((span, M), np.int64)
    for r in np.flatnonzero(last >= 0):
        m, ta = ev["req_model"][r], ev["req_t_arr_ms"][r]
        if not (0 <= ta <= first[r]):
            continue
        run[first[r]:last[r], m] += 1
        wait[ta:min(first[r], span), m] += 1
    np.testing.assert_array_equal(A_ms, run.reshape(K, win, M).sum(axis=1))
    np.testing.assert_array_equal(W_ms, wait.reshape(K, win, M).sum(axis=1))
