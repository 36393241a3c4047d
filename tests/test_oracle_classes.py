"""Pins for the per-(model, SLO class) mapping (Sec. II-A gives each model one
SLO class; with a class per request each (model, class) pair is scored as a
model of its own).

* a hand example, including ids outside the grid;
* one class is the identity on valid model ids;
* reducing the pairs and summing over classes gives the per-model reduction
  (the separately pinned reduce), and per-model SLO counts likewise.
"""
import numpy as np

import oracle
import tracegen


def test_hand_example():
    got = oracle.class_models([0, 2, 1, 3, -1, 1, 2], [1, 1, 0, 0, 0, 3, -1], 3, 3)
    assert got.tolist() == [1, 7, 3, -1, -1, -1, -1]


def test_one_class_is_the_identity_on_valid_ids():
    m = np.array([0, 4, 2, 7, 8, -2], np.int32)
    assert oracle.class_models(m, np.zeros(6, np.int32), 8, 1).tolist() == [0, 4, 2, 7, -1, -1]


def test_pairs_sum_to_models():
    w = tracegen.workload("mid", scale=0.02)
    req, M, win, K = w["requests"], w["M"], w["window_ms"], w["K"]
    rng = np.random.default_rng(3)
    n_cls = 3
    cls = rng.integers(0, n_cls, len(req["model"])).astype(np.int32)
    pair = dict(req, model=oracle.class_models(req["model"], cls, M, n_cls))
    per_pair = oracle.reduce_requests(pair, M * n_cls, win, K)
    per_model = oracle.reduce_requests(req, M, win, K)
    for a, b in zip(per_pair[:4], per_model[:4]):
        np.testing.assert_array_equal(a.reshape(K, M, n_cls).sum(axis=2), b)
    np.testing.assert_array_equal(per_pair[4], per_model[4])
    slo = np.asarray(w["slo_ttft_ms"], np.int32)
    na_p, nm_p = oracle.slo_counts_requests(pair, M * n_cls, win, K, np.repeat(slo, n_cls))
    na_m, nm_m = oracle.slo_counts_requests(req, M, win, K, slo)
    np.testing.assert_array_equal(na_p.reshape(K, M, n_cls).sum(axis=2), na_m)
    np.testing.assert_array_equal(nm_p.reshape(K, M, n_cls).sum(axis=2), nm_m)
