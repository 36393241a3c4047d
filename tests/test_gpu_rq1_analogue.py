"""The synthetic analogue of the paper's signal requirement (Sec. II-B) run
through the CUDA library: fixed-capacity segments of one model at five load
levels and three prefill/decode mixtures. Per mixture the five segments are
laid end to end as one trace (each shifted by the segment length), reduced,
calibrated and scored by the library, so theta is calibrated on the mixture's
pooled segments as a per-model profile would be (Sec. III-B). Checked: the
library's Z equals the oracle's on the same trace bit for bit; within a
mixture the mean Z of a segment falls strictly as its load rises; across all
segments the mean Z orders every pair whose TTFT attainment differs by at
least 0.05 the same way as attainment, but for at most one pair in twenty."""
import itertools

import numpy as np
import pytest

import oracle
from tests.test_rq1_analogue import KEYS, LOADS, MIXES, PROF, SLO_MS, WIN, K, _segment

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def segments():
    import torch
    import paper_2609_29160_gb300 as tre
    tre.load()
    torch.cuda.set_device(0)
    segs = {}
    for i, (rho, mix) in enumerate(itertools.product(LOADS, MIXES)):
        req = _segment(rho, mix, seed=700 + i)
        ttft = req["t_first_ms"].astype(np.int64) - req["t_arr_ms"]
        segs[(rho, mix)] = {"req": req, "health": float((ttft <= SLO_MS).mean())}
    KK = K * len(LOADS)
    for mix in MIXES:
        parts = []
        for j, rho in enumerate(LOADS):
            r = dict(segs[(rho, mix)]["req"])
            for k in ("t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms"):
                r[k] = (r[k] + j * K * WIN).astype(np.int32)
            parts.append(r)
        cat = {k: np.concatenate([p[k] for p in parts]) for k in KEYS}
        ref = oracle.pipeline_requests(cat, 1, WIN, KK, PROF, [SLO_MS], np.float64)
        dev = {k: torch.as_tensor(v).cuda() for k, v in cat.items()}
        c = tre.tss_window_reduce(1, WIN, KK, requests=dev)
        theta = tre.tss_calibrate(c, PROF, WIN, [SLO_MS], requests=dev, dtype="f64")
        sc = tre.tss_score(c, dict(PROF, theta=theta), WIN, dtype="f64")
        Z, cls = sc["Z"].cpu().numpy(), sc["cls"].cpu().numpy()
        np.testing.assert_array_equal(theta.cpu().numpy(), ref["theta"])
        np.testing.assert_array_equal(Z, ref["Z"])
        np.testing.assert_array_equal(cls, ref["cls"])
        for j, rho in enumerate(LOADS):
            z, k = Z[j * K:(j + 1) * K, 0], cls[j * K:(j + 1) * K, 0]
            segs[(rho, mix)]["mean_Z"] = float(z[k != oracle.IDLE].mean())
    return segs


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
