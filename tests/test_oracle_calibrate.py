"""Pins for the oracle's theta calibration (Sec. III-B: theta is the smallest
smoothed TSS value at which the SLO reliability target is still met).

Brute force: for every candidate value s, count directly the windows with
S >= s and how many of them are healthy; theta is the smallest qualifying s.
Plus monotonicity in the reliability target and the degenerate fallbacks.
"""
import numpy as np
import pytest

import oracle


def _brute_theta(S, cls, n_arr, n_met, ok_frac, rho):
    K, M = S.shape
    out, deg = [], 0
    for m in range(M):
        cand = [(S[k, m], n_met[k, m] >= ok_frac * n_arr[k, m]) for k in range(K)
                if cls[k, m] != oracle.IDLE and n_arr[k, m] >= 1 and S[k, m] > 0]
        if not cand:
            out.append(1.0)
            deg += 1
            continue
        ok = []
        for s, _ in cand:
            C = sum(1 for v, _ in cand if v >= s)
            H = sum(1 for v, h in cand if v >= s and h)
            if H >= rho * C:
                ok.append(s)
        if ok:
            out.append(min(ok))
        else:
            out.append(max(v for v, _ in cand))
            deg += 1
    return np.array(out), deg


def _rand_case(rng, K, M, n_levels=None, dtype=np.float64):
    if n_levels:
        S = rng.integers(1, n_levels + 1, (K, M)).astype(dtype) / 4
    else:
        S = rng.gamma(2.0, 3.0, (K, M)).astype(dtype)
    S[rng.random((K, M)) < 0.05] = 0
    cls = np.where(rng.random((K, M)) < 0.1, oracle.IDLE, oracle.NOM).astype(np.uint8)
    n_arr = rng.integers(0, 30, (K, M)).astype(np.int32)
    # healthier windows at higher S, with noise
    p_ok = np.clip(0.5 + S / (S.max() + 1e-9) * 0.6 + rng.normal(0, 0.15, (K, M)), 0, 1)
    n_met = rng.binomial(n_arr, p_ok).astype(np.int32)
    return S, cls, n_arr, n_met


@pytest.mark.parametrize("seed", range(6))
def test_theta_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    for dtype in (np.float64, np.float32):
        S, cls, n_arr, n_met = _rand_case(rng, 60, 3, n_levels=12 if seed % 2 else None, dtype=dtype)
        for rho in (0.5, 0.8, 0.95, 1.0):
            theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, rho)
            bt, bdeg = _brute_theta(S, cls, n_arr, n_met, 0.95, rho)
            np.testing.assert_array_equal(theta, bt.astype(dtype))
            assert deg == bdeg


def test_stricter_reliability_never_lowers_theta():
    rng = np.random.default_rng(11)
    S, cls, n_arr, n_met = _rand_case(rng, 400, 4)
    prev = None
    for rho in (0.3, 0.5, 0.7, 0.8, 0.9, 0.95, 0.99):
        theta, _ = oracle.calibrate(S, cls, n_arr, n_met, 0.9, rho)
        if prev is not None:
            assert (theta >= prev).all()
        prev = theta


def test_theta_separates_healthy_from_degraded():
    """Windows 31..100 healthy, 1..30 degraded. With S >= s for s <= 30 the
    healthy fraction is 70 / (101 - s): it reaches 0.95 first at s = 28
    (70/73 = 0.959; 70/74 = 0.946). At rho = 0.7 even s = 1 qualifies (70/100)."""
    K = 100
    S = np.arange(1, K + 1, dtype=np.float64).reshape(K, 1)
    cls = np.full((K, 1), oracle.NOM, np.uint8)
    n_arr = np.full((K, 1), 10, np.int32)
    n_met = np.where(S >= 31, 10, 3).astype(np.int32)
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, 0.95)
    assert theta[0] == 28.0 and deg == 0
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, 0.70)
    assert theta[0] == 1.0
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, 1.0)
    assert theta[0] == 31.0


def test_degenerate_fallbacks():
    S = np.array([[2.0, 0.0], [5.0, 0.0]])
    cls = np.array([[oracle.NOM, oracle.IDLE], [oracle.NOM, oracle.IDLE]], np.uint8)
    n_arr = np.array([[4, 3], [4, 3]], np.int32)
    n_met = np.array([[0, 3], [0, 3]], np.int32)
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, 0.95)
    # model 0: no healthy window -> max S; model 1: no candidate -> 1
    assert theta.tolist() == [5.0, 1.0] and deg == 2
