"""Pins for the oracle's window reduction: token counts (P, D) and gauges (A, W).

Each check ties the oracle to something other than itself: the hand-derived
worked example, the closed-form token staircase (a different formula from the
oracle's per-token enumeration), a brute-force membership count of the gauges,
conservation laws and the exact nesting of window lengths.
"""
import json
import os

import numpy as np
import pytest

import oracle
import tracegen
from tests.conftest import GOLDEN


def _w1():
    with open(os.path.join(GOLDEN, "w1_worked_example.json")) as f:
        return json.load(f)


def _rand_requests(rng, n, M, span_ms, max_lat_ms=4000, long_frac=0.05):
    t_arr = rng.integers(0, span_ms, n)
    wait = rng.integers(0, max_lat_ms, n) * (rng.random(n) < 0.5)
    pre = rng.integers(0, 800, n)
    dec = rng.integers(0, 3000, n)
    dec = np.where(rng.random(n) < long_frac, dec * 20, dec)
    L_out = rng.integers(1, 300, n)
    L_out = np.where(rng.random(n) < 0.1, 1, L_out)
    t_start = t_arr + wait
    t_first = t_start + pre
    t_end = np.where(L_out == 1, t_first, t_first + dec)
    return {"model": rng.integers(0, M, n).astype(np.int32),
            "t_arr_ms": t_arr.astype(np.int32), "t_start_ms": t_start.astype(np.int32),
            "t_first_ms": t_first.astype(np.int32), "t_end_ms": t_end.astype(np.int32),
            "L_in": rng.integers(0, 2000, n).astype(np.int32), "L_out": L_out.astype(np.int32)}


def _staircase_D(req, M, win, K):
    """Decode tokens per window from the closed-form count of tokens emitted
    strictly before T: 0 for T <= t_first, L_out for T > t_end, otherwise
    ceil((T - t_first)(L_out - 1) / (t_end - t_first))."""
    D = np.zeros((K, M), np.int64)
    for i in range(len(req["model"])):
        m = int(req["model"][i])
        tf, te, L = int(req["t_first_ms"][i]), int(req["t_end_ms"][i]), int(req["L_out"][i])

        def N(T):
            if T <= tf:
                return 0
            if T > te:
                return L
            if L == 1:
                return 1
            return -((-(T - tf) * (L - 1)) // (te - tf))

        for k in range(tf // win, min(K - 1, te // win) + 1):
            D[k, m] += N((k + 1) * win) - N(k * win)
    return D


def _brute_gauges(req, M, win, K):
    """A[k], W[k] by asking every request whether it is running / waiting at
    the last millisecond of window k."""
    A = np.zeros((K, M), np.int64)
    W = np.zeros((K, M), np.int64)
    last_ms = np.arange(K, dtype=np.int64) * win + (win - 1)
    for i in range(len(req["model"])):
        m = int(req["model"][i])
        ta, ts, te = int(req["t_arr_ms"][i]), int(req["t_start_ms"][i]), int(req["t_end_ms"][i])
        A[:, m] += (last_ms >= ts) & (last_ms < te)
        W[:, m] += (last_ms >= ta) & (last_ms < ts)
    return A, W


def test_worked_example_counts():
    g = _w1()
    req = {k: np.array(v, np.int32) for k, v in g["requests"].items()}
    P, D, A, W, drops = oracle.reduce_requests(req, 1, 1000, 3)
    e = g["expected"]
    assert P[:, 0].tolist() == e["P"]
    assert D[:, 0].tolist() == e["D"]
    assert A[:, 0].tolist() == e["A"]
    assert W[:, 0].tolist() == e["W"]
    assert drops.tolist() == [0, 0, 0]


@pytest.mark.parametrize("seed,win", [(1, 1000), (2, 100), (3, 250), (4, 7)])
def test_decode_tokens_match_closed_form_staircase(seed, win):
    rng = np.random.default_rng(seed)
    M, K = 3, 40
    req = _rand_requests(rng, 300, M, K * win * 3 // 4, max_lat_ms=max(50, 6 * win))
    _, D, _, _, _ = oracle.reduce_requests(req, M, win, K)
    np.testing.assert_array_equal(D, _staircase_D(req, M, win, K))


@pytest.mark.parametrize("seed,win", [(5, 1000), (6, 100), (7, 333)])
def test_gauges_match_brute_force_membership(seed, win):
    rng = np.random.default_rng(seed)
    M, K = 4, 50
    req = _rand_requests(rng, 400, M, K * win, max_lat_ms=30 * win)
    _, _, A, W, _ = oracle.reduce_requests(req, M, win, K)
    bA, bW = _brute_gauges(req, M, win, K)
    np.testing.assert_array_equal(A, bA)
    np.testing.assert_array_equal(W, bW)


def test_token_conservation_on_generated_trace():
    w = tracegen.workload("tiny", scale=0.3, seed=11)
    req, M, win, K = w["requests"], w["M"], w["window_ms"], w["K"]
    P, D, A, W, drops = oracle.reduce_requests(req, M, win, K)
    span = K * win
    for m in range(M):
        sel = req["model"] == m
        pin = sel & (req["t_first_ms"] < span)
        assert P[:, m].sum() == req["L_in"][pin].astype(np.int64).sum()
        done = sel & (req["t_end_ms"] < span)
        # every request that finished inside the trace contributes all its tokens;
        # unfinished ones contribute only what came before the end
        assert D[:, m].sum() >= req["L_out"][done].astype(np.int64).sum()
        assert D[:, m].sum() <= req["L_out"][sel].astype(np.int64).sum()
    assert (A >= 0).all() and (W >= 0).all()
    assert drops.tolist() == [0, 0, 0]


def test_prompt_tokens_by_bincount():
    rng = np.random.default_rng(9)
    M, win, K = 5, 200, 64
    req = _rand_requests(rng, 2000, M, K * win)
    P, _, _, _, _ = oracle.reduce_requests(req, M, win, K)
    span = K * win
    ok = req["t_first_ms"] < span
    idx = (req["t_first_ms"][ok] // win) * M + req["model"][ok]
    ref = np.bincount(idx, weights=req["L_in"][ok], minlength=K * M).reshape(K, M)
    np.testing.assert_array_equal(P, ref.astype(np.int64))


def test_drop_rules_and_precedence():
    # 0 ok, 1 bad model, 2 arrival past the end, 3 negative arrival,
    # 4 start before arrival, 5 end before first, 6 L_out = 0, 7 bad model AND late
    req = {
        "model":      np.array([0, 3, 0, 1, 1, 0, 0, -1], np.int32),
        "t_arr_ms":   np.array([10, 10, 5000, -1, 50, 10, 10, 9000], np.int32),
        "t_start_ms": np.array([20, 20, 5000, 0, 40, 20, 20, 9000], np.int32),
        "t_first_ms": np.array([30, 30, 5000, 0, 60, 30, 30, 9000], np.int32),
        "t_end_ms":   np.array([40, 40, 5000, 0, 70, 25, 40, 9000], np.int32),
        "L_in":       np.array([5, 5, 5, 5, 5, 5, 5, 5], np.int32),
        "L_out":      np.array([2, 2, 2, 2, 2, 2, 0, 2], np.int32),
    }
    P, D, A, W, drops = oracle.reduce_requests(req, 2, 1000, 4)
    # drops = [range, model, order]
    assert drops.tolist() == [2, 2, 3]
    assert P.sum() == 5 and D.sum() == 2


def test_empty_and_zero_windows():
    req = {k: np.zeros(0, np.int32) for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms",
                                               "t_end_ms", "L_in", "L_out")}
    P, D, A, W, drops = oracle.reduce_requests(req, 3, 1000, 5)
    assert P.shape == (5, 3) and not P.any() and not A.any()
    P, D, A, W, drops = oracle.reduce_requests(req, 3, 1000, 0)
    assert P.shape == (0, 3)


def test_nested_window_lengths_aggregate_exactly():
    """Counts at a window length that is a multiple q of a base length are the
    sums of q base windows; gauges are the base reading at sub-window (k+1)q-1."""
    w = tracegen.workload("tiny", scale=0.5, seed=5)
    req, M = w["requests"], w["M"]
    span = 600_000
    base = oracle.reduce_requests(req, M, 100, span // 100)
    for q in (5, 10, 20):
        P, D, A, W, _ = oracle.reduce_requests(req, M, 100 * q, span // (100 * q))
        Kq = span // (100 * q)
        np.testing.assert_array_equal(P, base[0].reshape(Kq, q, M).sum(1))
        np.testing.assert_array_equal(D, base[1].reshape(Kq, q, M).sum(1))
        np.testing.assert_array_equal(A, base[2][q - 1::q])
        np.testing.assert_array_equal(W, base[3][q - 1::q])


def _events_from_requests(req):
    """Token events placed exactly: one prompt token at t_start, the rest at
    t_first, decode tokens at their emission times (the last at t_end).
    Float seconds carry ms + 0.5 so the millisecond tick is unambiguous."""
    model, rid, t, ph = [], [], [], []
    for i in range(len(req["model"])):
        ts, tf, te = (int(req[k][i]) for k in ("t_start_ms", "t_first_ms", "t_end_ms"))
        L_in, L = int(req["L_in"][i]), int(req["L_out"][i])
        times = []
        if L_in >= 1:
            times += [(ts, 0)] + [(tf, 0)] * (L_in - 1)
        for j in range(L):
            times.append((tf if L == 1 else tf + (j * (te - tf)) // (L - 1), 1))
        for tt, p in times:
            model.append(int(req["model"][i]))
            rid.append(i)
            t.append((tt + 0.5) / 1000.0)
            ph.append(p)
    return {"model": np.array(model, np.int32), "req": np.array(rid, np.int32),
            "t_s": np.array(t, np.float32), "phase": np.array(ph, np.uint8),
            "req_model": req["model"].copy(), "req_t_arr_ms": req["t_arr_ms"].copy(),
            "req_ttft_ms": (req["t_first_ms"] - req["t_arr_ms"]).astype(np.int32)}


def test_events_agree_with_request_records():
    rng = np.random.default_rng(21)
    M, win, K = 3, 500, 40
    req = _rand_requests(rng, 150, M, K * win // 2, max_lat_ms=3000, long_frac=0.0)
    req["L_in"] = np.maximum(req["L_in"] % 40, 1).astype(np.int32)
    req["L_out"] = np.maximum(req["L_out"] % 30, 1).astype(np.int32)
    req["t_end_ms"] = np.where(req["L_out"] == 1, req["t_first_ms"], req["t_end_ms"]).astype(np.int32)
    ev = _events_from_requests(req)
    Pe, De, Ae, We, drops = oracle.reduce_events(ev, M, win, K)
    Pr, Dr, Ar, Wr, _ = oracle.reduce_requests(req, M, win, K)
    assert drops.tolist() == [0, 0, 0]
    # one prompt token sits at t_start instead of t_first
    adj = Pr.copy()
    for i in range(len(req["model"])):
        m = req["model"][i]
        adj[req["t_first_ms"][i] // win, m] -= 1
        adj[req["t_start_ms"][i] // win, m] += 1
    np.testing.assert_array_equal(Pe, adj)
    np.testing.assert_array_equal(De, Dr)
    np.testing.assert_array_equal(Ae, Ar)
    np.testing.assert_array_equal(We, Wr)
    na, nm = oracle.slo_counts_events(ev, M, win, K, np.array([1000, 3000, 500], np.int32))
    nra, nrm = oracle.slo_counts_requests(req, M, win, K, np.array([1000, 3000, 500], np.int32))
    np.testing.assert_array_equal(na, nra)
    np.testing.assert_array_equal(nm, nrm)


def test_event_drop_rules():
    ev = {"model": np.array([0, 1, 0, 0, 0, 2], np.int32),
          "req": np.array([0, 0, 0, 0, 5, 1], np.int32),
          "t_s": np.array([0.5, 0.5, -0.1, np.nan, 0.5, 0.7], np.float32),
          "phase": np.array([0, 1, 1, 1, 1, 3], np.uint8),
          "req_model": np.array([0, 2], np.int32), "req_t_arr_ms": np.array([100, 600], np.int32),
          "req_ttft_ms": np.array([10, 10], np.int32)}
    P, D, A, W, drops = oracle.reduce_events(ev, 3, 1000, 2)
    # [range, model, order]: event 1 (model != req_model), 4 (req out of table) -> model;
    # 2 (negative), 3 (NaN) -> range; 5 (phase 3) -> order
    assert drops.tolist() == [2, 2, 1]
    assert P[0, 0] == 1 and D.sum() == 0
