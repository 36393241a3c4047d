"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times (one marshalled pass of reduce -> calibrate -> normalize -> select
per trace, and the batched sweep), against the oracle on the same seeded
inputs, bit for bit: counts and drops, theta, S, Z, regions, receivers, moves
and final replicas.

Workloads (see the input recipe): three models over 600 s (fp64 and fp32);
eight models, 1M requests over one hour (fp32 and fp64); sixteen models with a
code/chat mix, 10M requests over 6 h at 500 ms windows; 64 models, ~200M token
events over 24 h at 100 ms windows; and the sweep of seven one-hour traces x 4
window lengths x 8 rescue thresholds x 8 pacing caps (1792 controller
instances), whose 28 (trace, window length) oracle units run in spawned worker
processes."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


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


def _oracle_path(w, dtype, events=None):
    """The oracle's whole path for one trace: counts, SLO counts, theta, S, Z,
    regions, receivers and the open-loop moves."""
    M, win, K = w["M"], w["window_ms"], w["K"]
    prof = tracegen.default_profile(M, win)
    if events is None:
        o = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], dtype)
    else:
        P, D, A, W, drops = oracle.reduce_events(events, M, win, K)
        n_arr, n_met = oracle.slo_counts_events(events, M, win, K, w["slo_ttft_ms"])
        S, _, cls, _ = oracle.score(P, D, A, W, prof, win, dtype)
        theta, deg = oracle.calibrate(S, cls, n_arr, n_met)
        p2 = dict(prof, theta=theta)
        S, Z, cls, recv = oracle.score(P, D, A, W, p2, win, dtype)
        o = {"P": P, "D": D, "A": A, "W": W, "drops": drops, "theta": theta, "degenerate": deg,
             "S": S, "Z": Z, "cls": cls, "recv": recv}
    mv, rf, _ = oracle.select_moves(o["Z"], o["cls"], 0.8, 1.2, win, w["budget"], w["r0"],
                                    w["r_min"], w["footprint"], w["fast_ms"], w["slow_ms"],
                                    w["pacing_cap"])
    o["moves"], o["r_final"] = mv, rf
    return o


def _run_plan(tre, w, dtype, events=None):
    M, win, K = w["M"], w["window_ms"], w["K"]
    prof = tracegen.default_profile(M, win)
    kw = {"events": _cuda(events)} if events is not None else {"requests": _cuda(w["requests"])}
    plan = tre.PipelinePlan(M, win, K, prof, w["slo_ttft_ms"], w["budget"], w["r0"], w["r_min"],
                            w["footprint"], dtype=dtype, fast_ms=w["fast_ms"],
                            slow_ms=w["slow_ms"], pacing_cap=w["pacing_cap"], moves_cap=1 << 16,
                            **kw)
    plan.run()
    return plan.results(), tre.read_diag(plan.diag)


def _compare(got, diag, ref):
    for k in ("P", "D", "A", "W", "theta", "S", "Z", "cls", "recv", "r_final"):
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)
    assert [diag["dropped_range"], diag["dropped_model"], diag["dropped_order"]] == \
        ref["drops"].tolist()
    assert got["n_moves"] == len(ref["moves"])
    f = ("window", "recv", "donor", "kind", "seq")
    g = np.stack([got["moves"][x].astype(np.int32) for x in f], 1)
    r = np.stack([ref["moves"][x] for x in f], 1)
    np.testing.assert_array_equal(g, r)


@pytest.mark.parametrize("name,dtype", [("tiny", "f64"), ("tiny", "f32"), ("mid", "f32"),
                                        ("mid", "f64"), ("hetero", "f32")])
def test_full_size_request_workloads(tre, name, dtype):
    w = tracegen.workload(name, scale=1.0)
    npdt = np.float32 if dtype == "f32" else np.float64
    ref = _oracle_path(w, npdt)
    got, diag = _run_plan(tre, w, dtype)
    _compare(got, diag, ref)
    assert len(ref["moves"]) > 0


def test_full_size_token_event_stream(tre):
    w = tracegen.workload("stream", scale=1.0)
    ev = w["events"]
    assert len(ev["model"]) > 150_000_000
    ref = _oracle_path(w, np.float32, events=ev)
    got, diag = _run_plan(tre, w, "f32", events=ev)
    _compare(got, diag, ref)
    assert len(ref["moves"]) > 0


# ---- the sweep at full size: 28 oracle units over spawned workers ----------
def _sweep_unit(args):
    ti, wi = args
    import numpy as np
    import oracle
    import tracegen
    # trace ti of the seven is the first trace of the sweep seeded at 100 + ti
    sw = tracegen.sweep_workload(scale=1.0, n_traces=1, seed0=100 + ti)
    win = int(sw["window_ms"][wi])
    alpha = min(1.0, win / 5000.0)
    ref = oracle.sweep([sw["traces"][0]], sw["M"], sw["duration_ms"], [win], sw["tau_crit"],
                       sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"], [alpha],
                       sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"], sw["footprint"],
                       dtype=np.float32)
    s = ref["series"][0]
    return ti, wi, {k: s[k] for k in ("P", "D", "A", "W", "S", "Z", "theta")}, \
        [(i["moves"], i["r_final"]) for i in ref["instances"]]


def test_full_size_sweep(tre):
    import multiprocessing as mp
    import os

    import torch
    sw = tracegen.sweep_workload(scale=1.0, n_traces=7)
    n_tr, n_w = len(sw["traces"]), len(sw["window_ms"])
    units = [(t, w) for t in range(n_tr) for w in range(n_w)]
    with mp.get_context("spawn").Pool(min(len(units), max(1, os.cpu_count() or 1))) as pool:
        res = pool.map_async(_sweep_unit, units, chunksize=1)
        alpha = [min(1.0, w / 5000.0) for w in sw["window_ms"]]
        moves_cap = 512
        out = tre.tre_sweep([_cuda(t) for t in sw["traces"]], sw["M"], sw["duration_ms"],
                            sw["window_ms"], alpha, sw["tau_crit"], sw["pacing_cap"], sw["w_p"],
                            sw["w_q"], sw["tau_surplus"], sw["slo_ttft_ms"], sw["budget"],
                            sw["r0"], sw["r_min"], sw["footprint"], dtype="f32",
                            moves_cap=moves_cap, want_counts=True, want_S=True)
        torch.cuda.synchronize()
        host = {k: out[k].cpu().numpy() for k in ("P", "D", "A", "W", "S", "Z")}
        theta = out["theta"].cpu().numpy()
        n_inst = n_tr * n_w * len(sw["tau_crit"]) * len(sw["pacing_cap"])
        moves = tre.sweep_moves(out, n_inst, moves_cap)
        n_moves = out["n_moves"].cpu().numpy()
        rf = out["r_final"].cpu().numpy()
        results = res.get(timeout=1200)
    M = sw["M"]
    K = [sw["duration_ms"] // int(x) for x in sw["window_ms"]]
    per_series = len(sw["tau_crit"]) * len(sw["pacing_cap"])
    f = ("window", "recv", "donor", "kind", "seq")
    checked = 0
    for ti, wi, s, inst in results:
        si = ti * n_w + wi
        off = sum(K[j % n_w] * M for j in range(si))
        n = K[wi] * M
        for k in ("P", "D", "A", "W", "S", "Z"):
            np.testing.assert_array_equal(host[k][off: off + n].reshape(K[wi], M), s[k],
                                          err_msg=f"series {si} {k}")
        np.testing.assert_array_equal(theta[si], s["theta"], err_msg=f"theta {si}")
        for j, (om, orf) in enumerate(inst):
            i = si * per_series + j
            np.testing.assert_array_equal(rf[i], orf, err_msg=f"instance {i}")
            assert int(n_moves[i]) == len(om), f"instance {i}"
            assert len(om) <= moves_cap
            if len(om):
                g = np.stack([moves[i][x].astype(np.int32) for x in f], 1)
                r = np.stack([om[x] for x in f], 1)
                np.testing.assert_array_equal(g, r, err_msg=f"instance {i}")
            checked += 1
    assert checked == n_inst == 1792
