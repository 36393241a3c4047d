"""Pins for the oracle's per-window ranking (Eq. 3 receiver, Sec. IV-B donor
acquisition order).

* hand windows: the order idle (by index), surplus (Z descending), nominal
  above the receiver (Z descending), critical models and the receiver left
  out, ties on Z by lower index, truncation to eight, all-idle windows;
* the walk: on a single control tick where every model holds one replica, no
  floor and no idle pool, the brute-force controller of test_oracle_select
  (a different formulation: smallest preference key over admissible pairs)
  releases donors in exactly this order.
"""
import numpy as np
import pytest

import oracle
from tests.test_oracle_select import _brute_walk

CRIT, NOM, SURP, IDLE = oracle.CRIT, oracle.NOM, oracle.SURP, oracle.IDLE


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_hand_window(dtype):
    # per-model thresholds: model 6 is critical at Z = 0.5 while model 8 is
    # nominal at 0.3, so the receiver (smallest Z, lowest index) is model 2
    Z = np.array([[0.9, 2.5, 0.3, 0.0, 1.7, 1.2, 0.5, 7.0, 0.3]], dtype)
    cls = np.array([[NOM, SURP, CRIT, IDLE, SURP, NOM, CRIT, IDLE, NOM]], np.uint8)
    recv, order = oracle.rank(Z, cls)
    assert recv.tolist() == [2]
    # idle 3, 7; surplus 1 (2.5), 4 (1.7); nominal above 0.3: 5 (1.2), 0 (0.9);
    # model 8 ties the receiver and is not above it; 6 is critical
    assert order.tolist() == [[3, 7, 1, 4, 5, 0, -1, -1]]


def test_ties_take_the_lower_index_and_idle_models_never_receive():
    Z = np.array([[1.5, 0.2, 1.5, 0.8, 0.8, 0.1]], np.float64)
    cls = np.array([[SURP, NOM, SURP, NOM, NOM, IDLE]], np.uint8)
    recv, order = oracle.rank(Z, cls)
    assert recv.tolist() == [1]                 # model 5 has the smallest Z but is idle
    assert order.tolist() == [[5, 0, 2, 3, 4, -1, -1, -1]]


def test_all_idle_and_single_model_windows():
    Z = np.array([[0.4, 0.9], [0.4, 0.9], [0.7, 0.7]], np.float32)
    cls = np.array([[IDLE, IDLE], [NOM, IDLE], [CRIT, CRIT]], np.uint8)
    recv, order = oracle.rank(Z, cls)
    assert recv.tolist() == [-1, 0, 0]
    assert order.tolist() == [[-1] * 8, [1] + [-1] * 7, [-1] * 8]
    recv, order = oracle.rank(np.array([[3.0]]), np.array([[SURP]], np.uint8))
    assert recv.tolist() == [0] and order.tolist() == [[-1] * 8]


def test_only_the_first_eight_donors_are_listed():
    M = 12
    Z = np.array([[0.2] + [1.0 + 0.1 * m for m in range(1, M)]], np.float64)
    cls = np.array([[CRIT] + [SURP] * (M - 1)], np.uint8)
    recv, order = oracle.rank(Z, cls)
    assert recv.tolist() == [0]
    assert order.tolist() == [list(range(11, 3, -1))]


@pytest.mark.parametrize("seed", range(6))
def test_order_is_the_walks_release_order(seed):
    rng = np.random.default_rng(seed)
    tc, ts = 0.6, 1.4
    vals = np.array([0.3, 0.5, 0.7, 0.8, 0.9, 1.0, 1.1, 1.2, 1.5, 2.0])
    checked = 0
    for _ in range(60):
        M = int(rng.integers(2, 12))
        z = rng.choice(vals, M)
        idle = rng.random(M) < 0.2
        if idle.all():
            idle[0] = False
        # the controller acts only when the lowest non-idle Z is below 1
        j = int(rng.choice(np.flatnonzero(~idle)))
        z[j] = min(z[j], 0.9)
        reg = np.where(idle, IDLE, np.where(z < tc, CRIT, np.where(z > ts, SURP, NOM)))
        Z, cls = z[None, :].astype(np.float64), reg[None, :].astype(np.uint8)
        recv, order = oracle.rank(Z, cls)
        # one window that ends both a fast and a slow tick; every model holds one
        # replica above a zero floor and the pool is empty, so each transition
        # releases the next donor in preference order
        moves, _ = _brute_walk(Z, cls, tc, ts, 10000, M, [1] * M, [0] * M, 5000, 10000, 8)
        donors = [mv[2] for mv in moves]
        want = [d for d in order[0].tolist() if d >= 0]
        assert donors == want
        assert {mv[1] for mv in moves} <= {int(recv[0])}
        checked += len(want) > 0
    assert checked >= 40
