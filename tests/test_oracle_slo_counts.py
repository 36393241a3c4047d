"""Pins for the oracle's SLO counts behind theta (Sec. III-B: theta is the lowest
smoothed TSS at which the SLO reliability target is still met; a request is
judged by its time to first token, counted in the window it arrived in).

The counts are pinned by a hand-derived fixture (tests/golden/slo_counts_hand.json)
whose requests sit exactly on the bound, wait in a queue before they start and
get their first token in a later window than their arrival, by an independent
NumPy statement of the rule on random records, and by a check that each
plausible misreading of the rule (strict comparison, TTFT measured from the
start of service, counting at the first-token window) changes the fixture's
expected counts, so the fixture would catch it.
"""
import json
import os

import numpy as np

import oracle
from tests.conftest import GOLDEN


def _fixture():
    with open(os.path.join(GOLDEN, "slo_counts_hand.json")) as f:
        return json.load(f)


def _req(fx):
    return {k: np.array(v, np.int32) for k, v in fx["requests"].items()}


def test_request_counts_match_the_hand_fixture():
    fx = _fixture()
    g = fx["grid"]
    n_arr, n_met = oracle.slo_counts_requests(_req(fx), g["n_models"], g["window_ms"],
                                              g["n_windows"], fx["slo_ttft_ms"])
    np.testing.assert_array_equal(n_arr, np.array(fx["expected"]["n_arr"]))
    np.testing.assert_array_equal(n_met, np.array(fx["expected"]["n_met"]))


def test_event_table_counts_match_the_hand_fixture():
    fx = _fixture()
    g = fx["grid"]
    ev = {k: np.array(v, np.int32) for k, v in fx["events_table"].items() if k != "note"}
    n_arr, n_met = oracle.slo_counts_events(ev, g["n_models"], g["window_ms"], g["n_windows"],
                                            fx["slo_ttft_ms"])
    np.testing.assert_array_equal(n_arr, np.array(fx["expected"]["n_arr"]))
    np.testing.assert_array_equal(n_met, np.array(fx["expected"]["n_met"]))


def _counts(req, M, win, K, slo, ttft_from="arrival", cmp="le", at="arrival"):
    """The counting rule in NumPy, with switches for the misreadings the
    fixture must reject."""
    m, ta, ts, tf, te = (req[k].astype(np.int64) for k in
                         ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms"))
    ok = ((m >= 0) & (m < M) & (ta >= 0) & (ta < K * win) & (ta <= ts) & (ts <= tf) &
          (tf <= te) & (req["L_in"] >= 0) & (req["L_out"] >= 1))
    m, ta, ts, tf = m[ok], ta[ok], ts[ok], tf[ok]
    ttft = tf - (ta if ttft_from == "arrival" else ts)
    bound = np.asarray(slo, np.int64)[m]
    met = ttft <= bound if cmp == "le" else ttft < bound
    k = (ta if at == "arrival" else tf) // win
    keep = k < K
    n_arr = np.zeros((K, M), np.int64)
    n_met = np.zeros((K, M), np.int64)
    np.add.at(n_arr, (k[keep], m[keep]), 1)
    np.add.at(n_met, (k[keep], m[keep]), met[keep].astype(np.int64))
    return n_arr, n_met


def test_numpy_statement_agrees_on_random_records():
    rng = np.random.default_rng(5)
    M, win, K, n = 5, 700, 60, 20000
    span = K * win
    ta = rng.integers(-win, span + win, n)
    ts = ta + rng.integers(0, 3000, n) * (rng.random(n) < 0.6)
    tf = ts + rng.integers(0, 2500, n)
    te = tf + rng.integers(0, 5000, n)
    bad = rng.random(n) < 0.02
    ts = np.where(bad, ta - 1, ts)
    req = {"model": rng.integers(-1, M + 1, n), "t_arr_ms": ta, "t_start_ms": ts,
           "t_first_ms": tf, "t_end_ms": te, "L_in": rng.integers(-1, 100, n),
           "L_out": rng.integers(0, 50, n)}
    req = {k: np.asarray(v, np.int32) for k, v in req.items()}
    slo = np.array([500, 1000, 1500, 2000, 700], np.int32)
    # bounds hit exactly by some requests
    hit = rng.random(n) < 0.1
    req["t_first_ms"] = np.where(hit & (req["model"] >= 0) & (req["model"] < M),
                                 req["t_arr_ms"] + slo[np.clip(req["model"], 0, M - 1)],
                                 req["t_first_ms"]).astype(np.int32)
    req["t_end_ms"] = np.maximum(req["t_end_ms"], req["t_first_ms"]).astype(np.int32)
    req["t_start_ms"] = np.minimum(req["t_start_ms"], req["t_first_ms"]).astype(np.int32)
    a_ref, m_ref = _counts(req, M, win, K, slo)
    n_arr, n_met = oracle.slo_counts_requests(req, M, win, K, slo)
    np.testing.assert_array_equal(n_arr, a_ref)
    np.testing.assert_array_equal(n_met, m_ref)
    assert n_met.sum() > 0 and n_met.sum() < n_arr.sum()


def test_fixture_rejects_each_misreading():
    fx = _fixture()
    g = fx["grid"]
    req = _req(fx)
    M, win, K = g["n_models"], g["window_ms"], g["n_windows"]
    want = (np.array(fx["expected"]["n_arr"]), np.array(fx["expected"]["n_met"]))
    same = _counts(req, M, win, K, fx["slo_ttft_ms"])
    assert all(np.array_equal(a, b) for a, b in zip(same, want))
    for kw in ({"cmp": "lt"}, {"ttft_from": "start"}, {"at": "first_token"}):
        got = _counts(req, M, win, K, fx["slo_ttft_ms"], **kw)
        assert not all(np.array_equal(a, b) for a, b in zip(got, want)), kw
