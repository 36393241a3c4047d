"""Pins for the oracle's Eq. 1 (raw TSS), EMA smoothing and Eq. 2 (Z, regions).

The pins: the paper's printed Fig. 1 pair and its ranking claim (Sec. II-B,
Sec. III-A), the meaning of Z (Sec. I, Sec. III-B), the demand floor
(Sec. II-B), the hand-derived worked example, the closed-form sum of the
exponential smoothing, and exact power-of-two scale invariance of Z.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
from tests.conftest import GOLDEN

PROFILE_KEYS = ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")


def _prof(**kw):
    p = {"w_p": 0.2, "w_q": 2.0, "alpha": 1.0, "theta": 1.0, "tau_crit": 0.8, "tau_surplus": 1.2}
    p.update(kw)
    return p


def _single_window(P, D, A, W, win, dtype=np.float64, **kw):
    a = lambda v: np.array([[v]], np.int32)
    return oracle.score(a(P), a(D), a(A), a(W), _prof(**kw), win, dtype)


def test_worked_example_values():
    with open(os.path.join(GOLDEN, "w1_worked_example.json")) as f:
        g = json.load(f)
    e = g["expected"]
    cnt = [np.array(e[k], np.int32).reshape(3, 1) for k in ("P", "D", "A", "W")]
    for dtype, rtol in ((np.float64, 1e-14), (np.float32, 2e-7)):
        S, Z, cls, recv = oracle.score(*cnt, g["profile"], 1000, dtype)
        for k in range(3):
            s = Fraction(e["S_num"][k], e["S_den"][k])
            assert S[k, 0] == pytest.approx(float(s), rel=rtol)
            assert Z[k, 0] == pytest.approx(float(s / 20), rel=rtol)
        assert cls[:, 0].tolist() == e["cls"]
        assert recv.tolist() == [0, 0, 0]


def _fig1():
    with open(os.path.join(GOLDEN, "fig1_pair.json")) as f:
        return json.load(f)


def _fig1_counts(case, scale5=True):
    """Realise the printed rates exactly: 10 s windows hold 10x the printed
    tokens/s as integers; running+waiting (printed to 0.1) times 5 is an
    integer, and scaling both denominators by 5 keeps their ordering."""
    P = int(round(case["prefill_tps"] * 10))
    D = int(round(case["decode_tps"] * 10))
    A = int(round(case["running_plus_waiting"] * 5))
    return P, D, A


@pytest.mark.parametrize("dtype", [np.float64, np.float32])
def test_fig1_pair_ranking_claim(dtype):
    g = _fig1()
    ph, dh = g["prefill_heavy"], g["decode_heavy"]
    # aggregate token throughput ranks the pair the wrong way (printed numbers)
    assert ph["prefill_tps"] + ph["decode_tps"] > dh["prefill_tps"] + dh["decode_tps"]
    Pp, Dp, Ap = _fig1_counts(ph)
    Pd, Dd, Ad = _fig1_counts(dh)

    def tss(P, D, A, w_p):
        S, _, _, _ = _single_window(P, D, A, 0, 10_000, dtype, w_p=w_p, w_q=1.0)
        return float(S[0, 0])

    # with a prefill weight below one, TSS ranks the SLO-violating
    # prefill-heavy case lower, as the paper states
    for w_p in (0.0, 0.1, 0.2, 0.22):
        assert tss(Pp, Dp, Ap, w_p) < tss(Pd, Dd, Ad, w_p)
    # the claim holds only below the crossover set by the printed numbers
    cross = (dh["decode_tps"] / dh["running_plus_waiting"] - ph["decode_tps"] / ph["running_plus_waiting"]) / (
        ph["prefill_tps"] / ph["running_plus_waiting"] - dh["prefill_tps"] / dh["running_plus_waiting"])
    assert 0.2296 < cross < 0.2297
    for w_p in (0.24, 0.5, 1.0):
        assert tss(Pp, Dp, Ap, w_p) > tss(Pd, Dd, Ad, w_p)


def test_z_meaning_half_service():
    """Z = 1 is the healthy boundary and 0.5 means half the needed per-request
    service (Sec. I, Sec. III-B)."""
    # 10 decode tokens in a 1 s window over 2 running requests: TSS = 5 tok/s/request
    S, Z, cls, _ = _single_window(0, 10, 2, 0, 1000, theta=10.0, alpha=1.0)
    assert S[0, 0] == 5.0 and Z[0, 0] == 0.5 and cls[0, 0] == oracle.CRIT
    S, Z, cls, _ = _single_window(0, 10, 2, 0, 1000, theta=5.0, alpha=1.0)
    assert Z[0, 0] == 1.0 and cls[0, 0] == oracle.NOM


def test_demand_floor():
    """Windows whose weighted demand is below one request divide by one (the
    'waiting-only raw inverse is 1.0' floor of Sec. II-B)."""
    for A, W, w_q in ((0, 0, 2.0), (0, 1, 0.5), (0, 1, 1.0)):
        S, _, cls, _ = _single_window(30, 7, A, W, 1000, w_q=w_q, w_p=0.5)
        assert S[0, 0] == 0.5 * 30 + 7
        assert cls[0, 0] != oracle.IDLE
    S, _, _, _ = _single_window(30, 7, 0, 3, 1000, w_q=2.0, w_p=0.5)
    assert S[0, 0] == (0.5 * 30 + 7) / 6


def test_idle_window_and_hold():
    P = np.array([[5], [0], [0], [3]], np.int32)
    Z0 = np.zeros_like(P)
    A = np.array([[1], [0], [0], [1]], np.int32)
    S, Z, cls, recv = oracle.score(P, Z0, A, Z0, _prof(alpha=0.5, w_p=1.0), 1000)
    assert cls[:, 0].tolist()[1:3] == [oracle.IDLE, oracle.IDLE]
    assert S[1, 0] == S[0, 0] == S[2, 0] == 5.0
    assert S[3, 0] == 0.5 * 3 + 0.5 * 5
    assert recv.tolist() == [0, -1, -1, 0]
    # a model that never had demand stays idle with S = 0
    S, Z, cls, recv = oracle.score(Z0, Z0, Z0, Z0, _prof(), 1000)
    assert (cls == oracle.IDLE).all() and not S.any() and (recv == -1).all()


def _closed_form_ema(raw, idle, alpha):
    """S_k = (1-a)^(k-k0) raw_{k0} + sum_{j in (k0, k]} a (1-a)^(n(j,k)) raw_j over
    non-idle windows j, where n(j, k) counts non-idle windows after j up to k."""
    out = np.zeros(len(raw))
    active = [j for j in range(len(raw)) if not idle[j]]
    for k in range(len(raw)):
        js = [j for j in active if j <= k]
        if not js:
            continue
        n = len(js)
        s = (1 - alpha) ** (n - 1) * raw[js[0]]
        for i, j in enumerate(js[1:], start=1):
            s += alpha * (1 - alpha) ** (n - 1 - i) * raw[j]
        out[k] = s
    return out


@pytest.mark.parametrize("alpha", [0.02, 0.3, 0.9])
def test_ema_matches_closed_form(alpha):
    rng = np.random.default_rng(int(alpha * 100))
    K = 120
    P = rng.integers(0, 500, (K, 1)).astype(np.int32)
    D = rng.integers(0, 200, (K, 1)).astype(np.int32)
    A = rng.integers(0, 20, (K, 1)).astype(np.int32)
    W = rng.integers(0, 20, (K, 1)).astype(np.int32)
    idle_rows = rng.random(K) < 0.2
    for a in (P, D, A, W):
        a[idle_rows] = 0
    idle_rows[:3] = True
    for a in (P, D, A, W):
        a[:3] = 0
    prof = _prof(alpha=alpha, w_p=0.3, w_q=1.5)
    raw = (0.3 * P[:, 0] + D[:, 0]) / np.maximum(A[:, 0] + 1.5 * W[:, 0], 1.0)
    S, _, _, _ = oracle.score(P, D, A, W, prof, 1000, np.float64)
    np.testing.assert_allclose(S[:, 0], _closed_form_ema(raw, idle_rows, alpha), rtol=1e-12, atol=0)


def test_alpha_one_and_constant_series():
    K = 50
    P = np.full((K, 1), 40, np.int32)
    D = np.full((K, 1), 9, np.int32)
    A = np.full((K, 1), 3, np.int32)
    W = np.full((K, 1), 1, np.int32)
    for alpha in (1.0, 0.37):
        S, _, _, _ = oracle.score(P, D, A, W, _prof(alpha=alpha), 1000, np.float64)
        raw = (0.2 * 40 + 9) / (3 + 2.0)
        # constant raw: S stays at raw up to one rounding of the affine step
        np.testing.assert_allclose(S[:, 0], raw, rtol=4e-16)
    rng = np.random.default_rng(3)
    P = rng.integers(0, 100, (K, 1)).astype(np.int32)
    S, _, _, _ = oracle.score(P, D, A, W, _prof(alpha=1.0), 1000, np.float64)
    np.testing.assert_array_equal(S[:, 0], (0.2 * (P[:, 0] / 1.0) + 9.0) / 5.0)


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_power_of_two_scale_invariance_of_z(dtype):
    """Scaling one model's token counts and its theta by 2^j leaves Z bit-exact,
    as does scaling its request counts by 2^j and theta by 2^-j: Z places
    models with different service scales on one comparable scale (Eq. 2)."""
    rng = np.random.default_rng(17)
    K = 200
    P = rng.integers(0, 2000, (K, 1)).astype(np.int32)
    D = rng.integers(0, 900, (K, 1)).astype(np.int32)
    A = rng.integers(1, 40, (K, 1)).astype(np.int32)
    W = rng.integers(0, 40, (K, 1)).astype(np.int32)
    prof = _prof(alpha=0.3, w_p=0.25, w_q=1.5, theta=3.0)
    _, Z0, c0, _ = oracle.score(P, D, A, W, prof, 500, dtype)
    for j in (1, 3, 6):
        _, Z1, c1, _ = oracle.score(P << j, D << j, A, W, dict(prof, theta=3.0 * 2 ** j), 500, dtype)
        np.testing.assert_array_equal(Z1, Z0)
        np.testing.assert_array_equal(c1, c0)
        _, Z2, c2, _ = oracle.score(P, D, A << j, W << j, dict(prof, theta=3.0 / 2 ** j), 500, dtype)
        np.testing.assert_array_equal(Z2, Z0)
        np.testing.assert_array_equal(c2, c0)


def test_regions_boundaries():
    # Z exactly at the thresholds is nominal; just beyond flips
    P = np.zeros((4, 1), np.int32)
    D = np.array([[8], [12], [7], [13]], np.int32)
    A = np.full((4, 1), 1, np.int32)
    S, Z, cls, _ = oracle.score(P, D, A, P, _prof(theta=10.0), 1000)
    assert Z[:, 0].tolist() == [0.8, 1.2, 0.7, 1.3]
    assert cls[:, 0].tolist() == [oracle.NOM, oracle.NOM, oracle.CRIT, oracle.SURP]


def test_receiver_is_argmin_over_non_idle_with_lowest_index_ties():
    P = np.zeros((3, 4), np.int32)
    D = np.array([[5, 3, 3, 0], [0, 0, 0, 0], [4, 9, 4, 1]], np.int32)
    A = np.array([[1, 1, 1, 0], [0, 0, 0, 0], [1, 1, 1, 0]], np.int32)
    S, Z, cls, recv = oracle.score(P, D, A, P, _prof(), 1000)
    assert recv.tolist() == [1, -1, 3]


def test_carry_splits_exactly():
    rng = np.random.default_rng(4)
    K, M = 300, 3
    cnt = [rng.integers(0, 50, (K, M)).astype(np.int32) * (rng.random((K, M)) < 0.7) for _ in range(4)]
    cnt = [c.astype(np.int32) for c in cnt]
    prof = _prof(alpha=0.1)
    for dtype in (np.float32, np.float64):
        S, Z, cls, recv = oracle.score(*cnt, prof, 100, dtype)
        carry = {"S": np.zeros(M, dtype), "init": np.zeros(M, np.uint8)}
        a = oracle.score(*[c[:137] for c in cnt], prof, 100, dtype, carry)
        b = oracle.score(*[c[137:] for c in cnt], prof, 100, dtype, carry)
        np.testing.assert_array_equal(np.concatenate([a[0], b[0]]), S)
        np.testing.assert_array_equal(np.concatenate([a[2], b[2]]), cls)
