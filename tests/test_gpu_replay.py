"""GPU parity of the closed-loop replay (Sec. IV-B controller acting on the
capacity that serves the requests it scores, Sec. IV-C bounded transfer,
Sec. VI-D actuation delays), called through the C ABI, against the oracle's
replay on the same latent requests, bit for bit: served records, the Z and
regions the controller saw, moves, final replicas, and the per-model counts of
served requests and of requests that met the TTFT bound."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu

REC = ("t_start_ms", "t_first_ms", "t_end_ms")
F = ("window", "recv", "donor", "kind", "seq")


@pytest.fixture(scope="module")
def tre():
    import torch
    import paper_2609_29160_gb300 as lib
    lib.load()
    torch.cuda.set_device(0)
    return lib


def _cuda(d):
    import torch
    return {k: torch.as_tensor(np.ascontiguousarray(v)).cuda() for k, v in d.items()}


def _mid_latent(scale, seed, duration_s):
    spec = tracegen.spec_mid(scale=scale, seed=seed, duration_s=duration_s)
    lat = tracegen.gen_latent(spec)
    return lat, 8, int(spec.budget)


def _counts(rec, lat, M, span, slo):
    """Served requests and requests meeting the TTFT bound per model, from the
    oracle's served records."""
    served = np.zeros(M, np.int64)
    met = np.zeros(M, np.int64)
    for m in range(M):
        sel = (lat["model"] == m) & (rec["t_start_ms"] >= 0)
        served[m] = int((rec["t_start_ms"][sel] < span).sum())
        ttft = rec["t_first_ms"][sel].astype(np.int64) - lat["t_arr_ms"][sel]
        met[m] = int((ttft <= slo[m]).sum())
    return served, met


def _check(tre, lat, M, win, K, prof, budget, r0, r_min, fp, dtype, settings, wake=0, sleep=0,
           slo=None, guard=None):
    """settings: list of (tau_crit, pacing_cap) per instance, as the replay
    orders them (thresholds outer, caps inner)."""
    taus = sorted({t for t, _ in settings}, key=[t for t, _ in settings].index)
    caps = sorted({c for _, c in settings}, key=[c for _, c in settings].index)
    slo = np.full(M, 1000, np.int32) if slo is None else slo
    out, moves, diag = tre.tre_replay(_cuda(lat), M, win, K, prof, budget, r0, r_min, fp,
                                      tau_list=taus, cap_list=caps, wake_ms=wake, sleep_ms=sleep,
                                      slo_ttft_ms=slo, guard_ttft_ms=guard, dtype=dtype,
                                      records=True, signal=True, moves_cap=1 << 14)
    npdt = np.float32 if dtype == "f32" else np.float64
    host = {k: v.cpu().numpy() for k, v in out.items() if k != "moves"}
    assert tre.read_diag(diag)["err"] == 0
    total = 0
    for i, (tau, cap) in enumerate((t, c) for t in taus for c in caps):
        ref = oracle.closed_loop(lat, M, win, K, prof, budget, r0, r_min, fp, tau,
                                 prof["tau_surplus"], pacing_cap=cap, dtype=npdt, wake_ms=wake,
                                 sleep_ms=sleep, guard_ms=guard)
        for k in REC:
            np.testing.assert_array_equal(host[k][i], ref["records"][k], err_msg=f"{i} {k}")
        np.testing.assert_array_equal(host["Z"][i], ref["Z"], err_msg=f"{i} Z")
        np.testing.assert_array_equal(host["cls"][i], ref["cls"], err_msg=f"{i} cls")
        np.testing.assert_array_equal(host["r_final"][i], ref["r_final"], err_msg=f"{i} r")
        assert int(host["n_moves"][i]) == len(ref["moves"]), i
        if len(ref["moves"]):
            g = np.stack([moves[i][x].astype(np.int32) for x in F], 1)
            r = np.stack([ref["moves"][x] for x in F], 1)
            np.testing.assert_array_equal(g, r, err_msg=f"{i} moves")
        served, met = _counts(ref["records"], lat, M, K * win, slo)
        np.testing.assert_array_equal(host["served"][i], served, err_msg=f"{i} served")
        np.testing.assert_array_equal(host["slo_met"][i], met, err_msg=f"{i} met")
        total += len(ref["moves"])
    return total


def _prof(M, theta=3.0):
    return {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": np.full(M, theta),
            "tau_crit": 0.8, "tau_surplus": 1.2}


@pytest.mark.parametrize("dtype", ["f64", "f32"])
@pytest.mark.parametrize("cap", [0, 1, 3])
def test_replay_matches_oracle(tre, dtype, cap):
    lat, M, budget = _mid_latent(0.01, 7, 900.0)
    K = 900
    n = _check(tre, lat, M, 1000, K, _prof(M), budget, lat["r0"], np.ones(M, np.int32),
               np.ones(M, np.int32), dtype, [(0.8, cap)])
    assert (n > 10) == (cap > 0)


@pytest.mark.parametrize("wake,sleep", [(1310, 1870), (0, 1870), (4000, 0), (4000, 3000)])
def test_replay_with_actuation_delays(tre, wake, sleep):
    """Delays longer than the rescue cadence also defer rescues behind
    rebalance transfers in progress."""
    lat, M, budget = _mid_latent(0.01, 8, 900.0)
    n = _check(tre, lat, M, 1000, 900, _prof(M), budget, lat["r0"], np.ones(M, np.int32),
               np.ones(M, np.int32), "f64", [(0.8, 2)], wake=wake, sleep=sleep)
    assert n > 10


@pytest.mark.parametrize("dtype", ["f64", "f32"])
@pytest.mark.parametrize("guard", [1500, 4000])
def test_replay_with_latency_guards(tre, dtype, guard):
    """Latency-guard breaches pre-empt rescue and hold donors; floors of zero
    let models lose their last routable replica."""
    lat, M, budget = _mid_latent(0.01, 13, 900.0)
    r_min = np.array([1, 0, 1, 0, 1, 0, 1, 0], np.int32)
    n = _check(tre, lat, M, 1000, 900, _prof(M), budget, lat["r0"], r_min, np.ones(M, np.int32),
               dtype, [(0.7, 1), (0.8, 2)], wake=1310, sleep=1870,
               guard=np.full(M, guard, np.int32))
    assert n > 10


def test_replay_batched_settings(tre):
    """Rescue thresholds x pacing caps side by side, one warp each, at 100 ms
    windows with delays."""
    lat, M, budget = _mid_latent(0.02, 9, 600.0)
    settings = [(t, c) for t in (0.5, 0.7, 0.8, 0.95) for c in (1, 2, 4)]
    slo = tracegen.slo_ttft_ms(M, 3)
    _check(tre, lat, M, 100, 6000, _prof(M), budget, lat["r0"], np.ones(M, np.int32),
           np.ones(M, np.int32), "f32", settings, wake=1310, sleep=1870, slo=slo,
           guard=2 * slo)


def test_replay_heterogeneous_footprints_and_pool(tre):
    lat, M, budget = _mid_latent(0.01, 10, 900.0)
    fp = np.array([1, 2, 1, 3, 1, 2, 1, 1], np.int32)
    r0 = np.maximum(lat["r0"] // fp, 1).astype(np.int32)
    budget = int((fp * r0).sum()) + 3
    r_min = np.array([1, 0, 1, 0, 1, 1, 0, 1], np.int32)
    _check(tre, lat, M, 1000, 900, _prof(M), budget, r0, r_min, fp, "f64", [(0.8, 3)],
           wake=500, sleep=700)


def test_replay_sixty_four_models_global_heaps(tre):
    """64 models (two per lane) with a 512-replica budget: the server heaps
    do not fit in shared memory and live in the workspace."""
    spec = tracegen.spec_stream(scale=0.05, seed=11, duration_s=1800.0)
    lat = tracegen.gen_latent(spec)
    M = spec.n_models
    prof = _prof(M, theta=2.0)
    _check(tre, lat, M, 100, 18000, prof, int(spec.budget), lat["r0"], np.ones(M, np.int32),
           np.ones(M, np.int32), "f32", [(0.8, 1), (0.8, 2)], wake=1310, sleep=1870,
           guard=np.full(M, 6000, np.int32))


def test_replay_invalid_records_are_not_served(tre):
    lat, M, budget = _mid_latent(0.005, 12, 600.0)
    lat = {k: (v.copy() if hasattr(v, "copy") else v) for k, v in lat.items()}
    n = len(lat["model"])
    rng = np.random.default_rng(3)
    idx = rng.choice(n, 60, replace=False)
    lat["model"][idx[:10]] = M
    lat["t_arr_ms"][idx[10:20]] = -5
    lat["t_arr_ms"][idx[20:30]] = 600 * 1000 + 7
    lat["d_first_ms"][idx[30:40]] = lat["d_total_ms"][idx[30:40]] + 1
    lat["L_out"][idx[40:50]] = 0
    lat["L_in"][idx[50:60]] = -1
    _check(tre, lat, M, 1000, 600, _prof(M), budget, lat["r0"], np.ones(M, np.int32),
           np.ones(M, np.int32), "f64", [(0.8, 1)], wake=100, sleep=100)
