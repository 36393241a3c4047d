"""Synthetic analogue of the paper's signal requirement (Sec. II-B): across
fixed-capacity trace segments that vary load intensity and prefill/decode
mixture, a signal fit for cross-model allocation ranks a segment as more
urgent when it faces more SLO-violation pressure.

Fifteen seeded segments of one model on four replicas (five utilisation levels
x three length mixtures, from the workload generator) are reduced, scored and
calibrated with the oracle; theta is calibrated per mixture on its own pooled
segments, as a per-model profile would be (Sec. III-B). Health is the share of
requests meeting a 5 s TTFT bound. Checked: within a mixture the mean Z falls
strictly as load rises, and across all segments the mean Z orders every pair
whose health differs by at least 0.05 the same way as health, but for at most
one pair in twenty. This is a property of the method on synthetic inputs, not
a parity pin.
"""
import itertools

import numpy as np
import pytest

import oracle
from tracegen import TraceSpec, gen_requests

KEYS = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")
MIXES = {"prefill-heavy": ((7.5, 0.8), (3.5, 0.8)), "balanced": ((6.0, 1.0), (5.0, 0.8)),
         "decode-heavy": ((4.0, 0.8), (6.2, 0.6))}
LOADS = (0.5, 0.7, 0.85, 0.95, 1.05)
WIN, K, SLO_MS = 1000, 900, 5000
PROF = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
        "tau_surplus": 1.2}


def _segment(rho, mix, seed):
    li, lo = MIXES[mix]
    spec = TraceSpec(n_models=1, duration_s=K * WIN / 1000.0, n_target=3000,
                     cost=np.array([1.0]), share=np.array([1.0]), len_in=np.array([li]),
                     len_out=np.array([lo]), budget=4, r0=np.array([4]), rho=rho,
                     rho_mode="max", seed=seed)
    req = gen_requests(spec)
    return {k: req[k] for k in KEYS}


@pytest.fixture(scope="module")
def segments():
    out = {}
    for i, (rho, mix) in enumerate(itertools.product(LOADS, MIXES)):
        req = _segment(rho, mix, seed=700 + i)
        P, D, A, W, _ = oracle.reduce_requests(req, 1, WIN, K)
        n_arr, n_met = oracle.slo_counts_requests(req, 1, WIN, K, [SLO_MS])
        ttft = req["t_first_ms"].astype(np.int64) - req["t_arr_ms"]
        out[(rho, mix)] = {"cnt": (P, D, A, W), "n_arr": n_arr, "n_met": n_met,
                           "health": float((ttft <= SLO_MS).mean())}
    # theta per mixture from its pooled segments
    for mix in MIXES:
        S_all, c_all, a_all, m_all = [], [], [], []
        for rho in LOADS:
            s = out[(rho, mix)]
            S, _, cls, _ = oracle.score(*s["cnt"], PROF, WIN, np.float64)
            S_all.append(S); c_all.append(cls); a_all.append(s["n_arr"]); m_all.append(s["n_met"])
        theta, _ = oracle.calibrate(np.concatenate(S_all), np.concatenate(c_all),
                                    np.concatenate(a_all), np.concatenate(m_all), 0.95, 0.95)
        for rho in LOADS:
            s = out[(rho, mix)]
            _, Z, cls, _ = oracle.score(*s["cnt"], dict(PROF, theta=theta), WIN, np.float64)
            busy = cls[:, 0] != oracle.IDLE
            s["mean_Z"] = float(Z[busy, 0].mean())
    return out


def test_health_falls_with_load(segments):
    for mix in MIXES:
        h = [segments[(rho, mix)]["health"] for rho in LOADS]
        assert h[0] == 1.0 and h[-1] < 0.5, (mix, h)


def test_z_falls_strictly_with_load_within_a_mixture(segments):
    for mix in MIXES:
        z = [segments[(rho, mix)]["mean_Z"] for rho in LOADS]
        assert all(a > b for a, b in zip(z, z[1:])), (mix, z)


def test_z_orders_segments_by_health(segments):
    agree = disagree = 0
    for a, b in itertools.combinations(segments.values(), 2):
        if abs(a["health"] - b["health"]) < 0.05:
            continue
        hi, lo = (a, b) if a["health"] > b["health"] else (b, a)
        if hi["mean_Z"] > lo["mean_Z"]:
            agree += 1
        else:
            disagree += 1
    assert agree >= 40
    assert disagree * 20 <= agree + disagree, (agree, disagree)
