"""Pins for the oracle's stage-aware signal (Sec. VIII: separate prefill and
decode states; Sec. III-A: prefill determines TTFT, decode TPOT).

* the running gauge splits at the first token: prefill + decode = the
  separately pinned running gauge, and a per-window brute force of the
  membership at the window's last millisecond gives each part;
* TPOT counts: a hand example and totals;
* reductions to the scalar signal: with no decode spans the prefill stage is
  the scalar signal with w_p = 1 and no decode tokens; with nothing waiting or
  prefilling the decode stage is the scalar signal without prompt tokens.
"""
import numpy as np
import pytest

import oracle
import tracegen

KEYS = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")


def _req(rng, n, M, win, K):
    ta = rng.integers(0, K * win, n)
    ts = ta + rng.integers(0, 3 * win, n)
    tf = ts + rng.integers(0, 2 * win, n)
    te = tf + rng.integers(0, 4 * win, n)
    L_out = rng.integers(1, 30, n)
    te = np.where(L_out == 1, tf, te)
    return {"model": rng.integers(0, M, n).astype(np.int32), "t_arr_ms": ta.astype(np.int32),
            "t_start_ms": ts.astype(np.int32), "t_first_ms": tf.astype(np.int32),
            "t_end_ms": te.astype(np.int32), "L_in": rng.integers(0, 90, n).astype(np.int32),
            "L_out": L_out.astype(np.int32)}


def _malformed(rng, req, M, win, K):
    """Some records the reduction drops: a start before the arrival, a first
    token before the start, an end before the first token, a bad model id, an
    arrival outside the grid, no output token."""
    req = {k: v.copy() for k, v in req.items()}
    n = len(req["model"])
    pick = rng.choice(n, 6 * (n // 10), replace=False).reshape(6, -1)
    req["t_start_ms"][pick[0]] = req["t_arr_ms"][pick[0]] - 1
    req["t_first_ms"][pick[1]] = req["t_start_ms"][pick[1]] - 1
    req["t_end_ms"][pick[2]] = req["t_first_ms"][pick[2]] - 1
    req["model"][pick[3]] = M
    req["t_arr_ms"][pick[4]] = K * win + 5
    req["L_out"][pick[5]] = 0
    return req


def _kept(req, M, win, K):
    m, ta, ts, tf, te = (req[k].astype(np.int64) for k in
                         ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms"))
    return ((m >= 0) & (m < M) & (ta >= 0) & (ta < K * win) & (ta <= ts) & (ts <= tf) &
            (tf <= te) & (req["L_in"] >= 0) & (req["L_out"] >= 1))


@pytest.mark.parametrize("seed,M,win,K", [(0, 3, 7, 20), (1, 2, 50, 12), (2, 4, 1, 60)])
@pytest.mark.parametrize("malformed", [False, True])
def test_running_gauge_splits_at_the_first_token(seed, M, win, K, malformed):
    rng = np.random.default_rng(seed)
    req = _req(rng, 80, M, win, K)
    if malformed:
        req = _malformed(rng, req, M, win, K)
    A_p, A_d = oracle.stage_gauges(req, M, win, K)
    A = oracle.reduce_requests(req, M, win, K)[2]
    np.testing.assert_array_equal(A_p + A_d, A)
    kept = _kept(req, M, win, K)
    for k in range(K):
        t = (k + 1) * win - 1                                    # last millisecond
        for m in range(M):
            sel = (req["model"] == m) & kept
            ts, tf, te = req["t_start_ms"][sel], req["t_first_ms"][sel], req["t_end_ms"][sel]
            assert A_p[k, m] == int(((ts <= t) & (t < tf)).sum())
            assert A_d[k, m] == int(((tf <= t) & (t < te)).sum())


def test_tpot_counts_hand_example():
    # window 1000 ms; model 0 bound 50 ms per token gap
    req = {"model": np.array([0, 0, 0, 0], np.int32),
           "t_arr_ms": np.array([10, 20, 1500, 30], np.int32),
           "t_start_ms": np.array([10, 20, 1500, 30], np.int32),
           "t_first_ms": np.array([100, 100, 1600, 40], np.int32),
           "t_end_ms": np.array([550, 551, 1600, 40], np.int32),
           "L_in": np.array([5, 5, 5, 5], np.int32),
           "L_out": np.array([10, 10, 1, 1], np.int32)}
    # request 0: 450 ms over 9 gaps = 50 ms, met; request 1: 451 ms, missed;
    # requests 2 and 3 have one output token and no gap
    n_dec, n_met = oracle.slo_tpot_counts_requests(req, 1, 1000, 2, [50])
    assert n_dec[:, 0].tolist() == [2, 0] and n_met[:, 0].tolist() == [1, 0]


def test_tpot_totals():
    w = tracegen.workload("mid", scale=0.01)
    req, M, win, K = w["requests"], w["M"], w["window_ms"], w["K"]
    n_dec, n_met = oracle.slo_tpot_counts_requests(req, M, win, K, np.full(M, 75))
    valid = (req["t_arr_ms"] < K * win) & (req["L_out"] > 1)
    assert n_dec.sum() == valid.sum()
    assert (n_met <= n_dec).all() and n_met.sum() > 0


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
def test_decode_stage_is_the_scalar_signal_without_queue_or_prefill(dtype):
    # requests that start and emit their first token on arrival, with no
    # prompt: nothing waits or prefills, so the running gauge is the decode
    # gauge and the scalar smoothed signal is the decode stage's
    rng = np.random.default_rng(9)
    M, win, K = 3, 100, 80
    req = _req(rng, 300, M, win, K)
    dec = dict(req, t_start_ms=req["t_arr_ms"], t_first_ms=req["t_arr_ms"],
               t_end_ms=np.maximum(req["t_end_ms"] - (req["t_first_ms"] - req["t_arr_ms"]),
                                   req["t_arr_ms"]).astype(np.int32),
               L_in=np.zeros_like(req["L_in"]))
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.3, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    st = oracle.stage_pipeline(dec, M, win, K, prof, np.full(M, 250), np.full(M, 40), dtype)
    P, D, A, W, _ = oracle.reduce_requests(dec, M, win, K)
    assert (P == 0).all() and (W == 0).all()
    np.testing.assert_array_equal(st["A_decode"], A)
    S_scalar = oracle.score(P, D, A, W, prof, win, dtype)[0]
    np.testing.assert_array_equal(st["decode"]["S"], S_scalar)


def test_hand_example():
    # one request, windows of 1 s: arrives at 0, starts at 200, first token at
    # 1500 (400 prompt tokens), 4 output tokens at 1500, 1600, 1700, 1800
    req = {"model": np.array([0], np.int32), "t_arr_ms": np.array([0], np.int32),
           "t_start_ms": np.array([200], np.int32), "t_first_ms": np.array([1500], np.int32),
           "t_end_ms": np.array([1800], np.int32), "L_in": np.array([400], np.int32),
           "L_out": np.array([4], np.int32)}
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.5, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    st = oracle.stage_pipeline(req, 1, 1000, 2, prof, [5000], [200], np.float64)
    # prefilling at 999 ms, neither at 1999 ms
    assert st["A_prefill"][:, 0].tolist() == [1, 0] and st["A_decode"][:, 0].tolist() == [0, 0]
    # prefill: window 0 raw 0 / 1 = 0, window 1 raw 400 / max(0, 1) = 400;
    # S = 0, then 0.5 * 400 + 0.5 * 0
    assert st["prefill"]["S"][:, 0].tolist() == [0.0, 200.0]
    # decode: window 0 idle (no tokens, nothing decoding), window 1 raw 4 / 1
    assert st["decode"]["cls"][0, 0] == oracle.IDLE
    assert st["decode"]["S"][1, 0] == 4.0
