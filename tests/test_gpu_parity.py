"""GPU parity: the CUDA library (called through the C ABI) against the CPU oracle
on the same seeded inputs. Integers, decisions and -- because the library
evaluates every floating-point step in the definition's order with one IEEE
rounding each -- the floating-point outputs too are compared bit for bit."""
import numpy as np
import pytest

import oracle
import tracegen

pytestmark = pytest.mark.gpu

REQ_KEYS = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")


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


def _np(t):
    return t.detach().cpu().numpy()


def _adversarial(rng, n, M, win, K):
    """Records on window boundaries, L_out = 1, zero-length spans, requests past
    the end, bad model ids, order violations, shuffled order."""
    span = K * win
    t_arr = rng.integers(-win, span + 2 * win, n)
    t_arr = np.where(rng.random(n) < 0.2, (t_arr // win) * win, t_arr)
    wait = rng.integers(0, 8 * win, n) * (rng.random(n) < 0.6)
    pre = rng.integers(0, 3 * win, n) * (rng.random(n) < 0.8)
    dec = rng.integers(0, 12 * win, n) * (rng.random(n) < 0.9)
    L_out = np.where(rng.random(n) < 0.15, 1, rng.integers(1, 600, n))
    t_start = t_arr + wait
    t_first = t_start + pre
    t_end = np.where(L_out == 1, t_first, t_first + dec)
    t_end = np.where(rng.random(n) < 0.05, (t_end // win) * win, t_end)
    model = rng.integers(0, M, n)
    model = np.where(rng.random(n) < 0.03, rng.choice([-1, M, M + 5], n), model)
    bad = rng.random(n) < 0.03
    t_start = np.where(bad, t_arr - 1, t_start)
    L_in = np.where(rng.random(n) < 0.01, -3, rng.integers(0, 4000, n))
    L_out = np.where(rng.random(n) < 0.01, 0, L_out)
    return {"model": model.astype(np.int32), "t_arr_ms": t_arr.astype(np.int32),
            "t_start_ms": t_start.astype(np.int32), "t_first_ms": t_first.astype(np.int32),
            "t_end_ms": t_end.astype(np.int32), "L_in": L_in.astype(np.int32),
            "L_out": L_out.astype(np.int32)}


def _check_reduce(tre, req, M, win, K):
    P, D, A, W, drops = oracle.reduce_requests(req, M, win, K)
    diag = tre.new_diag()
    c = tre.tss_window_reduce(M, win, K, requests=_cuda(req), diag=diag)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)
    d = tre.read_diag(diag)
    assert [d["dropped_range"], d["dropped_model"], d["dropped_order"]] == drops.tolist()
    return c


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("mid", 0.05), ("hetero", 0.01)])
def test_reduce_requests_generated(tre, name, scale):
    w = tracegen.workload(name, scale=scale)
    _check_reduce(tre, w["requests"], w["M"], w["window_ms"], w["K"])


@pytest.mark.parametrize("seed,M,win,K", [(1, 3, 1000, 50), (2, 8, 100, 700), (3, 17, 7, 333),
                                          (4, 64, 250, 40), (5, 1, 1, 5000)])
def test_reduce_requests_adversarial(tre, seed, M, win, K):
    rng = np.random.default_rng(seed)
    req = _adversarial(rng, 20000, M, win, K)
    _check_reduce(tre, req, M, win, K)
    # the same records shuffled give the same result
    perm = rng.permutation(len(req["model"]))
    _check_reduce(tre, {k: v[perm] for k, v in req.items()}, M, win, K)


def _sorted_long(rng, n, M, win, K):
    """Arrival-sorted records (the order telemetry arrives in) with queue waits,
    long decodes over many windows, very long outputs and some bad records."""
    span = K * win
    t_arr = np.sort(rng.integers(0, span + win, n))
    wait = rng.integers(0, 40 * win, n) * (rng.random(n) < 0.7)
    pre = rng.integers(0, 2 * win, n)
    dec = np.where(rng.random(n) < 0.3, rng.integers(0, 60 * win, n), rng.integers(0, 2 * win, n))
    L_out = np.where(rng.random(n) < 0.1, rng.integers(1, 100000, n), rng.integers(1, 400, n))
    t_start = t_arr + wait
    t_first = t_start + pre
    t_end = np.where(L_out == 1, t_first, t_first + dec)
    model = rng.integers(0, M, n)
    model = np.where(rng.random(n) < 0.01, M, model)
    return {"model": model.astype(np.int32), "t_arr_ms": t_arr.astype(np.int32),
            "t_start_ms": t_start.astype(np.int32), "t_first_ms": t_first.astype(np.int32),
            "t_end_ms": t_end.astype(np.int32),
            "L_in": rng.integers(0, 5000, n).astype(np.int32), "L_out": L_out.astype(np.int32)}


@pytest.mark.parametrize("seed,M,win,K,n", [(11, 8, 100, 3000, 60003), (12, 64, 50, 2000, 40001),
                                            (13, 5, 1000, 400, 9999)])
def test_reduce_requests_sorted_long_decodes(tre, seed, M, win, K, n):
    rng = np.random.default_rng(seed)
    _check_reduce(tre, _sorted_long(rng, n, M, win, K), M, win, K)


def test_reduce_requests_unaligned_columns(tre):
    """Columns that start 4 bytes past a 16-byte boundary take the scalar loads."""
    import torch
    rng = np.random.default_rng(21)
    M, win, K = 8, 100, 1500
    req = _sorted_long(rng, 30001, M, win, K)
    P, D, A, W, drops = oracle.reduce_requests(req, M, win, K)
    dev = {}
    for k, v in req.items():
        buf = torch.zeros(len(v) + 1, dtype=torch.int32, device="cuda")
        buf[1:] = torch.as_tensor(v).cuda()
        dev[k] = buf[1:]
        assert dev[k].data_ptr() % 16 == 4
    c = tre.tss_window_reduce(M, win, K, requests=dev)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)


def test_reduce_empty_and_zero_windows(tre):
    req = {k: np.zeros(0, np.int32) for k in REQ_KEYS}
    _check_reduce(tre, req, 4, 1000, 10)


def _events_case(seed, scale=0.002):
    w = tracegen.workload("stream", scale=scale, seed=seed)
    return w


def test_reduce_events(tre):
    w = _events_case(4)
    ev, M, win, K = w["events"], w["M"], w["window_ms"], w["K"]
    P, D, A, W, drops = oracle.reduce_events(ev, M, win, K)
    diag = tre.new_diag()
    c = tre.tss_window_reduce(M, win, K, events=_cuda(ev), diag=diag)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)
    d = tre.read_diag(diag)
    assert [d["dropped_range"], d["dropped_model"], d["dropped_order"]] == drops.tolist()


def test_reduce_events_shuffled_and_corrupt(tre):
    w = _events_case(5)
    ev = {k: v.copy() for k, v in w["events"].items()}
    M, win, K = w["M"], w["window_ms"], w["K"]
    rng = np.random.default_rng(0)
    n = len(ev["model"])
    idx = rng.choice(n, n // 50, replace=False)
    ev["t_s"][idx[: len(idx) // 4]] = np.float32(-1.0)
    ev["t_s"][idx[len(idx) // 4: len(idx) // 2]] = np.float32(np.nan)
    ev["phase"][idx[len(idx) // 2: 3 * len(idx) // 4]] = 7
    ev["model"][idx[3 * len(idx) // 4:]] = (ev["model"][idx[3 * len(idx) // 4:]] + 1) % M
    ev["t_s"][idx[:5]] = np.float32(-0.0)
    ev["req_t_arr_ms"][rng.choice(len(ev["req_model"]), 20)] = 10 ** 9
    perm = rng.permutation(n)
    ev = {k: (v[perm] if len(v) == n else v) for k, v in ev.items()}
    P, D, A, W, drops = oracle.reduce_events(ev, M, win, K)
    diag = tre.new_diag()
    c = tre.tss_window_reduce(M, win, K, events=_cuda(ev), diag=diag)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)
    d = tre.read_diag(diag)
    assert [d["dropped_range"], d["dropped_model"], d["dropped_order"]] == drops.tolist()


def _score_inputs(rng, K, M, idle_frac=0.2):
    cnt = {}
    for k, hi in (("P", 5000), ("D", 800), ("A", 30), ("W", 60)):
        cnt[k] = rng.integers(0, hi, (K, M)).astype(np.int32)
    idle = rng.random((K, M)) < idle_frac
    runs = rng.random(K) < 0.01               # long all-idle stretches
    idle |= np.repeat(runs, M).reshape(K, M)
    idle[: K // 20, M // 2:] = True           # some models start late
    for k in cnt:
        cnt[k][idle] = 0
    return cnt


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("K,M,win,alpha", [(600, 3, 1000, 0.2), (36000, 8, 100, 0.02),
                                           (43200, 16, 500, 0.1), (5000, 64, 100, 0.02),
                                           (3000, 5, 2000, 0.4), (257, 2, 100, 1.0)])
def test_score_bit_exact(tre, dtype, K, M, win, alpha):
    rng = np.random.default_rng(K + M)
    cnt = _score_inputs(rng, K, M)
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = {"w_p": rng.uniform(0.1, 0.3, M), "w_q": rng.uniform(1.0, 3.0, M),
            "alpha": np.full(M, alpha), "theta": rng.uniform(5, 50, M),
            "tau_crit": np.full(M, 0.8), "tau_surplus": np.full(M, 1.2)}
    S, Z, cls, recv = oracle.score(cnt["P"], cnt["D"], cnt["A"], cnt["W"], prof, win, npdt)
    diag = tre.new_diag()
    out = tre.tss_score(_cuda(cnt), prof, win, dtype=dtype, diag=diag)
    np.testing.assert_array_equal(_np(out["S"]), S)
    np.testing.assert_array_equal(_np(out["Z"]), Z)
    np.testing.assert_array_equal(_np(out["cls"]), cls)
    np.testing.assert_array_equal(_np(out["recv"]), recv)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_score_carry_across_calls(tre, dtype):
    import torch
    rng = np.random.default_rng(9)
    K, M, win = 20000, 6, 100
    cnt = _score_inputs(rng, K, M)
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.05, "theta": 10.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    S, Z, cls, _ = oracle.score(cnt["P"], cnt["D"], cnt["A"], cnt["W"], prof, win, npdt)
    tdt = torch.float32 if dtype == "f32" else torch.float64
    carry = {"S": torch.zeros(M, dtype=tdt, device="cuda"),
             "init": torch.zeros(M, dtype=torch.uint8, device="cuda")}
    parts = []
    for a, b in ((0, 7777), (7777, 7778), (7778, K)):
        sub = _cuda({k: v[a:b] for k, v in cnt.items()})
        parts.append(tre.tss_score(sub, prof, win, dtype=dtype, carry=carry))
    np.testing.assert_array_equal(np.concatenate([_np(p["S"]) for p in parts]), S)
    np.testing.assert_array_equal(np.concatenate([_np(p["cls"]) for p in parts]), cls)


def test_score_is_deterministic(tre):
    rng = np.random.default_rng(5)
    cnt = _cuda(_score_inputs(rng, 50000, 8))
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.02, "theta": 10.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    a = tre.tss_score(cnt, prof, 100)
    b = tre.tss_score(cnt, prof, 100)
    for k in ("S", "Z", "cls", "recv"):
        assert (a[k] == b[k]).all()


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("mid", 0.05), ("hetero", 0.005)])
def test_pipeline_requests(tre, dtype, name, scale):
    w = tracegen.workload(name, scale=scale)
    M, win, K = w["M"], w["window_ms"], w["K"]
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(M, win)
    o = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], npdt)
    req = _cuda(w["requests"])
    c = tre.tss_window_reduce(M, win, K, requests=req)
    diag = tre.new_diag()
    theta = tre.tss_calibrate(c, prof, win, w["slo_ttft_ms"], requests=req, dtype=dtype,
                              diag=diag)
    np.testing.assert_array_equal(_np(theta), o["theta"])
    assert tre.read_diag(diag)["degenerate_calib"] == o["degenerate"]
    sc = tre.tss_score(c, dict(prof, theta=theta), win, dtype=dtype)
    for k in ("S", "Z", "cls", "recv"):
        np.testing.assert_array_equal(_np(sc[k]), o[k], err_msg=k)
    rk = tre.tss_rank(sc["Z"], sc["cls"], win)
    orv, odn = oracle.rank(o["Z"], o["cls"])
    np.testing.assert_array_equal(_np(rk["recv"]), orv)
    np.testing.assert_array_equal(_np(rk["recv"]), o["recv"])
    np.testing.assert_array_equal(_np(rk["donors"]), odn)
    for cap in (1, 3):
        for tc in (0.6, 0.9):
            p2 = dict(prof, theta=theta, tau_crit=np.full(M, tc))
            mv, rf, n, _ = tre.tre_select_moves(sc["Z"], sc["cls"], p2, win, w["budget"],
                                                w["r0"], w["r_min"], w["footprint"],
                                                pacing_cap=cap)
            om, orf, _ = oracle.select_moves(o["Z"], o["cls"], tc, 1.2, win, w["budget"],
                                             w["r0"], w["r_min"], w["footprint"], pacing_cap=cap)
            assert n == len(om)
            np.testing.assert_array_equal(_np(rf), orf)
            got = np.stack([mv[f].astype(np.int32) for f in ("window", "recv", "donor", "kind",
                                                               "seq")], 1) if n else np.zeros((0, 5))
            ref = np.stack([om[f] for f in ("window", "recv", "donor", "kind", "seq")], 1) \
                if n else np.zeros((0, 5))
            np.testing.assert_array_equal(got, ref)


def _rank_case(rng, K, M, dtype):
    """Z drawn from a few values (ties on Z), every region, idle runs, and
    some all-idle windows."""
    vals = np.array([0.25, 0.5, 0.75, 0.9, 1.0, 1.1, 1.3, 2.0, 3.5], dtype)
    Z = rng.choice(vals, (K, M))
    cls = rng.choice(np.array([0, 1, 2, 3], np.uint8), (K, M), p=[0.2, 0.4, 0.25, 0.15])
    cls[rng.random(K) < 0.03] = 3
    return np.ascontiguousarray(Z), np.ascontiguousarray(cls)


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
@pytest.mark.parametrize("seed,K,M", [(31, 4099, 8), (32, 1037, 1), (33, 777, 5), (37, 301, 12),
                                      (38, 2000, 16), (39, 99, 17), (34, 513, 33), (35, 129, 100),
                                      (36, 17, 1024)])
def test_rank_matches_oracle(tre, dtype, seed, K, M):
    rng = np.random.default_rng(seed)
    Z, cls = _rank_case(rng, K, M, dtype)
    orv, odn = oracle.rank(Z, cls)
    g = tre.tss_rank(*_cuda({"Z": Z, "cls": cls}).values())
    np.testing.assert_array_equal(_np(g["recv"]), orv)
    np.testing.assert_array_equal(_np(g["donors"]), odn)
    # either output alone gives the same values
    only_r = tre.tss_rank(*_cuda({"Z": Z, "cls": cls}).values(), donors=False)
    only_d = tre.tss_rank(*_cuda({"Z": Z, "cls": cls}).values(), recv=False)
    assert only_r["donors"] is None and only_d["recv"] is None
    np.testing.assert_array_equal(_np(only_r["recv"]), orv)
    np.testing.assert_array_equal(_np(only_d["donors"]), odn)


def test_rank_empty_grid(tre):
    import torch
    g = tre.tss_rank(torch.zeros((0, 4), dtype=torch.float32, device="cuda"),
                     torch.zeros((0, 4), dtype=torch.uint8, device="cuda"))
    assert g["recv"].numel() == 0 and g["donors"].shape == (0, 8)


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("mid", 0.05), ("hetero", 0.01)])
def test_mean_occupancy_reduce_generated(tre, name, scale):
    w = tracegen.workload(name, scale=scale)
    M, win, K = w["M"], w["window_ms"], w["K"]
    A_ms, W_ms = oracle.occupancy_mean_requests(w["requests"], M, win, K)
    c = tre.tss_window_reduce(M, win, K, requests=_cuda(w["requests"]), mean_occupancy=True)
    np.testing.assert_array_equal(_np(c["A_ms"]), A_ms)
    np.testing.assert_array_equal(_np(c["W_ms"]), W_ms)
    P, D, A, W, _ = oracle.reduce_requests(w["requests"], M, win, K)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)


@pytest.mark.parametrize("seed,M,win,K", [(41, 3, 1000, 50), (42, 8, 100, 700), (43, 17, 7, 333),
                                          (44, 64, 250, 40), (45, 1, 1, 5000)])
def test_mean_occupancy_reduce_adversarial(tre, seed, M, win, K):
    rng = np.random.default_rng(seed)
    req = _adversarial(rng, 20000, M, win, K)
    A_ms, W_ms = oracle.occupancy_mean_requests(req, M, win, K)
    diag = tre.new_diag()
    c = tre.tss_window_reduce(M, win, K, requests=_cuda(req), diag=diag, mean_occupancy=True)
    np.testing.assert_array_equal(_np(c["A_ms"]), A_ms)
    np.testing.assert_array_equal(_np(c["W_ms"]), W_ms)
    _, _, _, _, drops = oracle.reduce_requests(req, M, win, K)
    d = tre.read_diag(diag)   # drops are counted once, by the reduction
    assert [d["dropped_range"], d["dropped_model"], d["dropped_order"]] == drops.tolist()


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("mid", 0.05)])
def test_mean_occupancy_pipeline(tre, dtype, name, scale):
    w = tracegen.workload(name, scale=scale)
    M, win, K = w["M"], w["window_ms"], w["K"]
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(M, win)
    o = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], npdt,
                                 mean_occupancy=True)
    req = _cuda(w["requests"])
    c = tre.tss_window_reduce(M, win, K, requests=req, mean_occupancy=True)
    diag = tre.new_diag()
    theta = tre.tss_calibrate(c, prof, win, w["slo_ttft_ms"], requests=req, dtype=dtype,
                              diag=diag)
    np.testing.assert_array_equal(_np(theta), o["theta"])
    sc = tre.tss_score(c, dict(prof, theta=theta), win, dtype=dtype)
    for k in ("S", "Z", "cls", "recv"):
        np.testing.assert_array_equal(_np(sc[k]), o[k], err_msg=k)
    # the sampled gauges give a different score on this workload
    plain = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], npdt)
    assert not np.array_equal(plain["S"], o["S"])


def test_mean_occupancy_empty_and_refusals(tre):
    import torch
    M, win, K = 4, 100, 30
    empty = {k: torch.zeros(0, dtype=torch.int32, device="cuda") for k in REQ_KEYS}
    c = tre.tss_window_reduce(M, win, K, requests=empty, mean_occupancy=True)
    assert int(c["A_ms"].abs().sum()) == 0 and int(c["W_ms"].abs().sum()) == 0
    ev = {"model": torch.zeros(0, dtype=torch.int32, device="cuda"),
          "req": torch.zeros(0, dtype=torch.int32, device="cuda"),
          "t_s": torch.zeros(0, dtype=torch.float32, device="cuda"),
          "phase": torch.zeros(0, dtype=torch.uint8, device="cuda"),
          "req_model": torch.zeros(3, dtype=torch.int32, device="cuda"),
          "req_t_arr_ms": torch.zeros(3, dtype=torch.int32, device="cuda"),
          "req_ttft_ms": torch.zeros(3, dtype=torch.int32, device="cuda")}
    c = tre.tss_window_reduce(M, win, K, events=ev, mean_occupancy=True)
    assert int(c["A_ms"].abs().sum()) == 0 and int(c["W_ms"].abs().sum()) == 0


def _corrupt_events(ev, rng, M):
    ev = {k: v.copy() for k, v in ev.items()}
    n = len(ev["model"])
    idx = rng.choice(n, n // 50, replace=False)
    q = len(idx) // 4
    ev["t_s"][idx[:q]] = np.float32(-1.0)
    ev["t_s"][idx[q: 2 * q]] = np.float32(np.nan)
    ev["phase"][idx[2 * q: 3 * q]] = 7
    ev["model"][idx[3 * q:]] = (ev["model"][idx[3 * q:]] + 1) % M
    ev["req_t_arr_ms"][rng.choice(len(ev["req_model"]), 20)] = 10 ** 9
    perm = rng.permutation(n)
    for k in ("model", "req", "t_s", "phase"):
        ev[k] = ev[k][perm]
    return ev


@pytest.mark.parametrize("seed,corrupt", [(7, False), (8, True)])
def test_mean_occupancy_token_events(tre, seed, corrupt):
    """Time-averaged occupancy from token events (running from a request's first
    to its last valid event, waiting from its arrival to its first), on a
    time-sorted stream and on a shuffled stream with corrupt events."""
    w = _events_case(seed)
    ev, M, win, K = w["events"], w["M"], w["window_ms"], w["K"]
    if corrupt:
        ev = _corrupt_events(ev, np.random.default_rng(seed), M)
    A_ms, W_ms = oracle.occupancy_mean_events(ev, M, win, K)
    c = tre.tss_window_reduce(M, win, K, events=_cuda(ev), mean_occupancy=True)
    np.testing.assert_array_equal(_np(c["A_ms"]), A_ms)
    np.testing.assert_array_equal(_np(c["W_ms"]), W_ms)
    P, D, A, W, _ = oracle.reduce_events(ev, M, win, K)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_mean_occupancy_token_events_pipeline(tre, dtype):
    """Calibration and scoring with the event-form window means in Eq. 1's
    demand term."""
    w = _events_case(9)
    ev, M, win, K = w["events"], w["M"], w["window_ms"], w["K"]
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(M, win)
    P, D, A, W, _ = oracle.reduce_events(ev, M, win, K)
    occ = oracle.occupancy_mean_events(ev, M, win, K)
    n_arr, n_met = oracle.slo_counts_events(ev, M, win, K, w["slo_ttft_ms"])
    S, _, cls, _ = oracle.score(P, D, A, W, prof, win, npdt, occ_ms=occ)
    theta, _ = oracle.calibrate(S, cls, n_arr, n_met)
    S, Z, cls, recv = oracle.score(P, D, A, W, dict(prof, theta=theta), win, npdt, occ_ms=occ)
    evc = _cuda(ev)
    c = tre.tss_window_reduce(M, win, K, events=evc, mean_occupancy=True)
    th = tre.tss_calibrate(c, prof, win, w["slo_ttft_ms"], events=evc, dtype=dtype)
    np.testing.assert_array_equal(_np(th), theta)
    sc = tre.tss_score(c, dict(prof, theta=th), win, dtype=dtype)
    for k, ref in (("S", S), ("Z", Z), ("cls", cls), ("recv", recv)):
        np.testing.assert_array_equal(_np(sc[k]), ref, err_msg=k)


def test_class_models_mapping(tre):
    import torch
    rng = np.random.default_rng(51)
    n, M, n_cls = 100003, 8, 3
    model = rng.integers(-2, M + 2, n).astype(np.int32)
    cls = rng.integers(-1, n_cls + 1, n).astype(np.int32)
    got = tre.tss_class_models(torch.as_tensor(model).cuda(), torch.as_tensor(cls).cuda(), M,
                               n_cls)
    np.testing.assert_array_equal(_np(got), oracle.class_models(model, cls, M, n_cls))


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_per_class_pipeline(tre, dtype):
    # one SLO class per request: each (model, class) pair is scored as a model
    w = tracegen.workload("mid", scale=0.05)
    M, win, K = w["M"], w["window_ms"], w["K"]
    n_cls = 3
    rng = np.random.default_rng(52)
    cls = rng.integers(0, n_cls, len(w["requests"]["model"])).astype(np.int32)
    pair_model = oracle.class_models(w["requests"]["model"], cls, M, n_cls)
    pair_req = dict(w["requests"], model=pair_model)
    Mp = M * n_cls
    slo = np.tile(np.array(tracegen.SLO_CLASSES_MS, np.int32), M)
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(Mp, win)
    o = oracle.pipeline_requests(pair_req, Mp, win, K, prof, slo, npdt)
    req = _cuda(w["requests"])
    import torch
    req["model"] = tre.tss_class_models(req["model"], torch.as_tensor(cls).cuda(), M, n_cls)
    np.testing.assert_array_equal(_np(req["model"]), pair_model)
    c = tre.tss_window_reduce(Mp, win, K, requests=req)
    for k in "PDAW":
        np.testing.assert_array_equal(_np(c[k]), o[k], err_msg=k)
    theta = tre.tss_calibrate(c, prof, win, slo, requests=req, dtype=dtype)
    np.testing.assert_array_equal(_np(theta), o["theta"])
    sc = tre.tss_score(c, dict(prof, theta=theta), win, dtype=dtype)
    for k in ("S", "Z", "cls", "recv"):
        np.testing.assert_array_equal(_np(sc[k]), o[k], err_msg=k)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_stage_signal(tre, dtype):
    w = tracegen.workload("mid", scale=0.02)
    M, win, K = w["M"], w["window_ms"], w["K"]
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(M, win)
    tpot = np.full(M, 60, np.int32)
    o = oracle.stage_pipeline(w["requests"], M, win, K, prof, w["slo_ttft_ms"], tpot, npdt)
    req = _cuda(w["requests"])
    A_p, A_d = tre.tss_stage_gauges(M, win, K, req)
    np.testing.assert_array_equal(_np(A_p), o["A_prefill"])
    np.testing.assert_array_equal(_np(A_d), o["A_decode"])
    c = tre.tss_window_reduce(M, win, K, requests=req)
    diag = tre.new_diag()
    theta_p, theta_d = tre.tss_stage_calibrate(c, A_p, A_d, prof, win, w["slo_ttft_ms"], tpot,
                                               req, dtype=dtype, diag=diag)
    np.testing.assert_array_equal(_np(theta_p), o["prefill"]["theta"])
    np.testing.assert_array_equal(_np(theta_d), o["decode"]["theta"])
    assert tre.read_diag(diag)["degenerate_calib"] == \
        o["prefill"]["degenerate"] + o["decode"]["degenerate"]
    sp, sd = tre.tss_stage_score(c, A_p, A_d, prof, win, theta_p, theta_d, dtype=dtype)
    for k in ("S", "Z", "cls"):
        np.testing.assert_array_equal(_np(sp[k]), o["prefill"][k], err_msg="prefill " + k)
        np.testing.assert_array_equal(_np(sd[k]), o["decode"][k], err_msg="decode " + k)


@pytest.mark.parametrize("seed,M,win,K", [(41, 5, 1000, 120), (42, 64, 100, 900)])
def test_stage_signal_adversarial(tre, seed, M, win, K):
    """Records on window boundaries, one output token (no TPOT count), spans
    past the grid, bad ids and order violations; TPOT bounds hit exactly."""
    rng = np.random.default_rng(seed)
    req = _adversarial(rng, 30000, M, win, K)
    tpot = rng.integers(1, 40, M).astype(np.int32)
    ok = (req["L_out"] > 1) & (rng.random(len(req["L_out"])) < 0.2)
    te = req["t_first_ms"].astype(np.int64) + tpot[np.clip(req["model"], 0, M - 1)].astype(
        np.int64) * (req["L_out"].astype(np.int64) - 1)
    req["t_end_ms"] = np.where(ok & (te < 2 ** 31 - 1), te, req["t_end_ms"]).astype(np.int32)
    slo = rng.integers(100, 3000, M).astype(np.int32)
    prof = tracegen.default_profile(M, win)
    for dtype, npdt in (("f32", np.float32), ("f64", np.float64)):
        o = oracle.stage_pipeline(req, M, win, K, prof, slo, tpot, npdt)
        rc = _cuda(req)
        A_p, A_d = tre.tss_stage_gauges(M, win, K, rc)
        np.testing.assert_array_equal(_np(A_p), o["A_prefill"])
        np.testing.assert_array_equal(_np(A_d), o["A_decode"])
        c = tre.tss_window_reduce(M, win, K, requests=rc)
        th_p, th_d = tre.tss_stage_calibrate(c, A_p, A_d, prof, win, slo, tpot, rc, dtype=dtype)
        np.testing.assert_array_equal(_np(th_p), o["prefill"]["theta"])
        np.testing.assert_array_equal(_np(th_d), o["decode"]["theta"])
        sp, sd = tre.tss_stage_score(c, A_p, A_d, prof, win, th_p, th_d, dtype=dtype)
        for k in ("S", "Z", "cls"):
            np.testing.assert_array_equal(_np(sp[k]), o["prefill"][k], err_msg="prefill " + k)
            np.testing.assert_array_equal(_np(sd[k]), o["decode"][k], err_msg="decode " + k)


def test_calibrate_events(tre):
    w = _events_case(6)
    ev, M, win, K = w["events"], w["M"], w["window_ms"], w["K"]
    prof = tracegen.default_profile(M, win)
    P, D, A, W, _ = oracle.reduce_events(ev, M, win, K)
    n_arr, n_met = oracle.slo_counts_events(ev, M, win, K, w["slo_ttft_ms"])
    S, _, cls, _ = oracle.score(P, D, A, W, prof, win, np.float32)
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met)
    evc = _cuda(ev)
    c = tre.tss_window_reduce(M, win, K, events=evc)
    diag = tre.new_diag()
    th = tre.tss_calibrate(c, prof, win, w["slo_ttft_ms"], events=evc, dtype="f32", diag=diag)
    np.testing.assert_array_equal(_np(th), theta)
    assert tre.read_diag(diag)["degenerate_calib"] == deg


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_calibrate_adversarial_ties(tre, dtype):
    """Few distinct S levels (many exact ties), idle and zero-S windows, rho 1."""
    import torch
    rng = np.random.default_rng(3)
    K, M, win = 3000, 5, 1000
    cnt = _score_inputs(rng, K, M, idle_frac=0.3)
    cnt["P"] = (cnt["P"] // 1000 * 1000).astype(np.int32)
    cnt["D"] = (cnt["D"] // 200 * 200).astype(np.int32)
    cnt["A"] = np.where(cnt["A"] > 0, 4, 0).astype(np.int32)
    cnt["W"] = np.zeros_like(cnt["W"])
    prof = {"w_p": 0.25, "w_q": 2.0, "alpha": 1.0, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    npdt = np.float32 if dtype == "f32" else np.float64
    S, _, cls, _ = oracle.score(cnt["P"], cnt["D"], cnt["A"], cnt["W"], prof, win, npdt)
    # arrivals: one request per window at a random ms; met with probability rising in S
    req = {k: [] for k in REQ_KEYS}
    for k in range(K):
        for m in range(M):
            if rng.random() < 0.7:
                ta = k * win + int(rng.integers(0, win))
                ok = rng.random() < min(1.0, 0.3 + S[k, m] / (S.max() + 1e-9))
                tf = ta + (100 if ok else 5000)
                for key, v in zip(REQ_KEYS, (m, ta, ta, tf, tf, 1, 1)):
                    req[key].append(v)
    req = {k: np.array(v, np.int32) for k, v in req.items()}
    slo = np.full(M, 1000, np.int32)
    n_arr, n_met = oracle.slo_counts_requests(req, M, win, K, slo)
    for rho in (0.5, 0.95, 1.0):
        theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, rho)
        diag = tre.new_diag()
        th = tre.tss_calibrate(_cuda(cnt), prof, win, slo, requests=_cuda(req), dtype=dtype,
                               ok_frac=0.95, reliability=rho, diag=diag)
        np.testing.assert_array_equal(_np(th), theta)
        assert tre.read_diag(diag)["degenerate_calib"] == deg
    # the same records shuffled (arrival windows no longer in runs), and with
    # records out of range at the head of every slice of 4096: the same theta
    perm = rng.permutation(len(req["model"]))
    shuf = {k: v[perm] for k, v in req.items()}
    heads = np.arange(0, len(perm), 4096)
    shuf["t_arr_ms"][heads] = K * win + 5
    n_arr, n_met = oracle.slo_counts_requests(shuf, M, win, K, slo)
    theta, deg = oracle.calibrate(S, cls, n_arr, n_met, 0.95, 0.95)
    for order in (shuf, {k: v[np.argsort(shuf["t_arr_ms"], kind="stable")] for k, v in shuf.items()}):
        th = tre.tss_calibrate(_cuda(cnt), prof, win, slo, requests=_cuda(order), dtype=dtype,
                               ok_frac=0.95, reliability=0.95)
        np.testing.assert_array_equal(_np(th), theta)


def test_select_heterogeneous_footprints_and_overflow(tre):
    import torch
    rng = np.random.default_rng(12)
    K, M, win = 3000, 6, 1000
    Z = rng.choice(np.array([0.3, 0.6, 0.85, 0.95, 1.0, 1.1, 1.3, 2.0]), (K, M)).astype(np.float32)
    cls = np.where(rng.random((K, M)) < 0.1, oracle.IDLE, oracle.NOM).astype(np.uint8)
    g = np.array([1, 2, 3, 1, 2, 1], np.int32)
    r0 = np.array([3, 2, 2, 4, 1, 3], np.int32)
    budget = int((g * r0).sum()) + 2
    r_min = np.array([1, 1, 0, 2, 0, 1], np.int32)
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    om, orf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, budget, r0, r_min, g, 5000, 10000, 3)
    Zc, Cc = torch.as_tensor(Z).cuda(), torch.as_tensor(cls).cuda()
    mv, rf, n, diag = tre.tre_select_moves(Zc, Cc, prof, win, budget, r0, r_min, g, pacing_cap=3,
                                           moves_cap=len(om) + 5)
    assert n == len(om)
    np.testing.assert_array_equal(_np(rf), orf)
    for a, b in zip(mv, om):
        assert (int(a["window"]), int(a["recv"]), int(a["donor"]), int(a["kind"]),
                int(a["seq"])) == tuple(int(x) for x in b)
    assert tre.read_diag(diag)["err"] == 0
    # overflow: only the first `cap` moves are written, the count is the full one
    mv, rf, n, diag = tre.tre_select_moves(Zc, Cc, prof, win, budget, r0, r_min, g, pacing_cap=3,
                                           moves_cap=7)
    assert n == len(om) and len(mv) == 7
    assert tre.read_diag(diag)["err"] == 4
    np.testing.assert_array_equal(_np(rf), orf)


@pytest.mark.parametrize("M,r_each,extra", [(8, 20, 3), (8, 40, 5), (5, 60, 0), (7, 1, 1)])
@pytest.mark.parametrize("cap", [1, 2])
def test_select_unit_footprints_small_and_large_budgets(tre, M, r_each, extra, cap):
    # budgets up to 255 keep every model's replicas in one byte; larger ones not
    import torch
    rng = np.random.default_rng(M * 100 + r_each)
    K, win = 4000, 500
    Z = rng.choice(np.array([0.3, 0.6, 0.85, 0.95, 1.0, 1.1, 1.3, 2.0]), (K, M)).astype(np.float32)
    cls = np.where(rng.random((K, M)) < 0.1, oracle.IDLE, oracle.NOM).astype(np.uint8)
    g = np.ones(M, np.int32)
    r0 = np.full(M, r_each, np.int32)
    r0[0] = 0
    budget = int(r0.sum()) + extra
    r_min = np.where(np.arange(M) % 3 == 1, 1, 0).astype(np.int32)
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    om, orf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, budget, r0, r_min, g, 5000, 10000, cap)
    Zc, Cc = torch.as_tensor(Z).cuda(), torch.as_tensor(cls).cuda()
    mv, rf, n, diag = tre.tre_select_moves(Zc, Cc, prof, win, budget, r0, r_min, g,
                                           pacing_cap=cap, moves_cap=len(om) + 5)
    assert n == len(om) and n > 0
    np.testing.assert_array_equal(_np(rf), orf)
    got = np.stack([mv[f].astype(np.int32) for f in ("window", "recv", "donor", "kind", "seq")], 1)
    ref = np.stack([om[f] for f in ("window", "recv", "donor", "kind", "seq")], 1)
    np.testing.assert_array_equal(got, ref)
    assert tre.read_diag(diag)["err"] == 0


@pytest.mark.parametrize("cap", [1, 3])
def test_select_and_rank_on_threshold_values_and_ties(tre, cap):
    # Z exactly at tau_crit (0.8), tau_surplus (1.2) and the rebalance bound (1),
    # with ties across models: every comparison is strict on both sides
    import torch
    rng = np.random.default_rng(61 + cap)
    K, M, win = 3000, 6, 1000
    Z = rng.choice(np.array([0.5, 0.8, 0.8, 1.0, 1.0, 1.2, 1.2, 1.5]), (K, M)).astype(np.float32)
    cls = np.where(rng.random((K, M)) < 0.1, oracle.IDLE, oracle.NOM).astype(np.uint8)
    r0 = np.array([3, 2, 2, 4, 1, 3], np.int32)
    budget = int(r0.sum()) + 1
    r_min = np.array([1, 0, 1, 0, 0, 1], np.int32)
    g = np.ones(M, np.int32)
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    om, orf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, budget, r0, r_min, g, 5000, 10000,
                                     cap)
    Zc, Cc = torch.as_tensor(Z).cuda(), torch.as_tensor(cls).cuda()
    mv, rf, n, _ = tre.tre_select_moves(Zc, Cc, prof, win, budget, r0, r_min, g,
                                        pacing_cap=cap, moves_cap=len(om) + 5)
    assert n == len(om) and n > 0
    np.testing.assert_array_equal(_np(rf), orf)
    got = np.stack([mv[f].astype(np.int32) for f in ("window", "recv", "donor", "kind", "seq")], 1)
    ref = np.stack([om[f] for f in ("window", "recv", "donor", "kind", "seq")], 1)
    np.testing.assert_array_equal(got, ref)
    # the per-window ranking on classes from the same thresholds
    reg = np.where(cls == oracle.IDLE, oracle.IDLE,
                   np.where(Z < np.float32(0.8), oracle.CRIT,
                            np.where(Z > np.float32(1.2), oracle.SURP, oracle.NOM))).astype(np.uint8)
    orv, odn = oracle.rank(Z, reg)
    rk = tre.tss_rank(Zc, torch.as_tensor(reg).cuda(), win)
    np.testing.assert_array_equal(_np(rk["recv"]), orv)
    np.testing.assert_array_equal(_np(rk["donors"]), odn)


def _sweep_case(scale, n_traces, duration_s):
    sw = tracegen.sweep_workload(scale=scale, n_traces=n_traces, duration_s=duration_s)
    alpha = [min(1.0, w / 5000.0) for w in sw["window_ms"]]
    return sw, alpha


def _run_sweep_both(tre, sw, alpha, moves_cap, dtype="f32"):
    M = sw["M"]
    npdt = np.float32 if dtype == "f32" else np.float64
    ref = oracle.sweep(sw["traces"], M, sw["duration_ms"], sw["window_ms"], sw["tau_crit"],
                       sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"], alpha,
                       sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"], sw["footprint"],
                       dtype=npdt)
    out = tre.tre_sweep([_cuda(t) for t in sw["traces"]], M, sw["duration_ms"], sw["window_ms"],
                        alpha, sw["tau_crit"], sw["pacing_cap"], sw["w_p"], sw["w_q"],
                        sw["tau_surplus"], sw["slo_ttft_ms"], sw["budget"], sw["r0"],
                        sw["r_min"], sw["footprint"], dtype=dtype, moves_cap=moves_cap,
                        want_counts=True, want_S=True)
    return ref, out


def _compare_sweep(tre, sw, ref, out, moves_cap):
    M = sw["M"]
    off = 0
    theta = _np(out["theta"])
    for si, s in enumerate(ref["series"]):
        n = s["K"] * M
        for k in ("P", "D", "A", "W", "S", "Z"):
            np.testing.assert_array_equal(_np(out[k][off: off + n]).reshape(s["K"], M), s[k],
                                          err_msg=f"series {si} {k}")
        np.testing.assert_array_equal(theta[si], s["theta"], err_msg=f"theta {si}")
        off += n
    n_inst = len(ref["instances"])
    moves = tre.sweep_moves(out, n_inst, moves_cap)
    rf = _np(out["r_final"])
    for i, inst in enumerate(ref["instances"]):
        np.testing.assert_array_equal(rf[i], inst["r_final"], err_msg=f"instance {i}")
        got = moves[i]
        om = inst["moves"]
        assert int(_np(out["n_moves"])[i]) == len(om), f"instance {i}"
        assert len(got) == min(len(om), moves_cap)
        for a, b in zip(got, om):
            assert (int(a["window"]), int(a["recv"]), int(a["donor"]), int(a["kind"]),
                    int(a["seq"])) == tuple(int(x) for x in b), f"instance {i}"


def test_sweep_small(tre):
    sw, alpha = _sweep_case(0.02, 2, 600.0)
    sw["tau_crit"] = sw["tau_crit"][::3]
    sw["pacing_cap"] = sw["pacing_cap"][::3]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512)
    _compare_sweep(tre, sw, ref, out, 512)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_sweep_many_series_rank_in_walk(tre, dtype):
    """Five traces x 4 window lengths x 8 rescue thresholds: at least one
    (series, threshold) block per SM, so the jump walk ranks its own ticks
    from the Z and class rows (one launch) instead of reading tick tables."""
    sw, alpha = _sweep_case(0.02, 5, 600.0)
    sw["pacing_cap"] = sw["pacing_cap"][::4]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512, dtype=dtype)
    _compare_sweep(tre, sw, ref, out, 512)


def test_reduce_requests_from_pinned_host_memory(tre):
    """Record columns left in pinned host memory that the GPU addresses
    directly give the same counts as device-resident columns."""
    import torch
    rng = np.random.default_rng(31)
    M, win, K = 8, 100, 1200
    req = _sorted_long(rng, 20001, M, win, K)
    host = {k: torch.as_tensor(v).pin_memory() for k, v in req.items()}
    ref = tre.tss_window_reduce(M, win, K, requests=_cuda(req))
    got = tre.tss_window_reduce(M, win, K, requests=host)
    for k in "PDAW":
        assert torch.equal(got[k], ref[k]), k


@pytest.mark.parametrize("where", ["device", "pinned_host", "mixed"])
def test_reduce_requests_1024_models(tre, where):
    """The largest model count the library takes: the staging leaves less room
    per CTA, and records read from host memory are copied into shared memory
    beside it (fewer records per CTA). `mixed` leaves one column in host
    memory."""
    import torch
    rng = np.random.default_rng(1024)
    M, win, K = 1024, 100, 600
    req = _adversarial(rng, 120000, M, win, K)
    P, D, A, W, drops = oracle.reduce_requests(req, M, win, K)
    if where == "device":
        cols = _cuda(req)
    elif where == "pinned_host":
        cols = {k: torch.as_tensor(v).pin_memory() for k, v in req.items()}
    else:
        cols = _cuda(req)
        cols["L_out"] = torch.as_tensor(req["L_out"]).pin_memory()
    diag = tre.new_diag()
    c = tre.tss_window_reduce(M, win, K, requests=cols, diag=diag)
    for k, ref in zip("PDAW", (P, D, A, W)):
        np.testing.assert_array_equal(_np(c[k]), ref, err_msg=k)
    d = tre.read_diag(diag)
    assert [d["dropped_range"], d["dropped_model"], d["dropped_order"]] == drops.tolist()


def test_calibrate_1024_models(tre):
    import torch
    rng = np.random.default_rng(4)
    M, win, K = 1024, 1000, 300
    req = _adversarial(rng, 150000, M, win, K)
    slo = rng.integers(200, 3000, M).astype(np.int32)
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    o = oracle.pipeline_requests(req, M, win, K, prof, slo, np.float32)
    rc = _cuda(req)
    c = tre.tss_window_reduce(M, win, K, requests=rc)
    th = tre.tss_calibrate(c, prof, win, slo, requests=rc, dtype="f32")
    np.testing.assert_array_equal(_np(th), o["theta"])


def test_reduce_refuses_pageable_host_columns(tre):
    """Record columns in ordinary (pageable) host memory would fault a kernel
    reading them: the call refuses them before launching anything."""
    import ctypes as C
    import torch
    cols = {k: torch.zeros(64, dtype=torch.int32) for k in REQ_KEYS}   # not pinned
    lib = tre.load()
    g = tre.Grid(4, 100, 10)
    rq = tre.requests_struct(cols)
    P, D, A, W = (torch.empty((10, 4), dtype=torch.int32, device="cuda") for _ in range(4))
    out = tre.Counts(P.data_ptr(), D.data_ptr(), A.data_ptr(), W.data_ptr())
    size = C.c_size_t(0)
    st = lib.tss_window_reduce(C.byref(g), C.byref(rq), None, out, None, C.byref(size), None, None)
    assert st == 1      # TRE_EINVAL


def test_sweep_f64(tre):
    sw, alpha = _sweep_case(0.02, 2, 600.0)
    sw["tau_crit"] = sw["tau_crit"][1::3]
    sw["pacing_cap"] = sw["pacing_cap"][1::3]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512, dtype="f64")
    _compare_sweep(tre, sw, ref, out, 512)


def test_sweep_refuses_window_lengths_not_multiples_of_the_shortest(tre):
    """Every window length must be a multiple of the shortest one (the grid
    the records are reduced on); 200/300/600 ms is refused."""
    sw, _ = _sweep_case(0.01, 1, 600.0)
    sw["window_ms"] = np.array([200, 300, 600], dtype=np.int32)
    alpha = [min(1.0, w / 5000.0) for w in sw["window_ms"]]
    with pytest.raises(tre.TreError) as ei:
        tre.tre_sweep([_cuda(t) for t in sw["traces"]], sw["M"], sw["duration_ms"],
                      sw["window_ms"], alpha, sw["tau_crit"], sw["pacing_cap"], sw["w_p"],
                      sw["w_q"], sw["tau_surplus"], sw["slo_ttft_ms"], sw["budget"], sw["r0"],
                      sw["r_min"], sw["footprint"])
    assert ei.value.code == 1


def test_sweep_more_window_lengths_than_the_fused_pass_takes(tre):
    """Nine window lengths: the gauge scan and the coarsening run as separate
    passes."""
    sw, _ = _sweep_case(0.01, 1, 600.0)
    sw["window_ms"] = np.array([100, 200, 300, 400, 500, 600, 1000, 1200, 2000], dtype=np.int32)
    alpha = [min(1.0, w / 5000.0) for w in sw["window_ms"]]
    sw["tau_crit"] = sw["tau_crit"][::4]
    sw["pacing_cap"] = sw["pacing_cap"][::4]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512)
    _compare_sweep(tre, sw, ref, out, 512)


def test_sweep_heterogeneous_footprints(tre):
    """Models of different replica footprints: the walk's general transition
    path (a receiver may need several donor releases)."""
    sw, alpha = _sweep_case(0.02, 1, 600.0)
    M = sw["M"]
    sw["footprint"] = np.array([1, 2, 1, 3, 1, 2, 1, 1][:M], dtype=np.int32)
    sw["budget"] = int((sw["footprint"] * sw["r0"]).sum()) + 3
    sw["tau_crit"] = sw["tau_crit"][::2]
    sw["pacing_cap"] = sw["pacing_cap"][::3]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512)
    _compare_sweep(tre, sw, ref, out, 512)


def test_sweep_twelve_models(tre):
    """More than eight models: the walk's 16-model tables and donor scan."""
    sw, alpha = _sweep_case(0.02, 1, 600.0)
    rng = np.random.default_rng(5)
    M0 = sw["M"]
    for t in sw["traces"]:
        t["model"] = np.where(rng.random(len(t["model"])) < 0.35, t["model"] + M0,
                              t["model"]).astype(np.int32)
        t["model"] = np.minimum(t["model"], 11).astype(np.int32)
    M = 12
    ext = lambda a: np.concatenate([np.asarray(a), np.asarray(a)])[:M]
    sw["M"] = M
    for k in ("w_p", "w_q", "tau_surplus", "slo_ttft_ms", "r0", "r_min", "footprint"):
        if np.ndim(sw[k]):
            sw[k] = ext(sw[k]).astype(np.asarray(sw[k]).dtype)
    sw["budget"] = int(sw["r0"].sum()) + 2
    sw["tau_crit"] = sw["tau_crit"][::3]
    sw["pacing_cap"] = sw["pacing_cap"][::3]
    ref, out = _run_sweep_both(tre, sw, alpha, moves_cap=512)
    _compare_sweep(tre, sw, ref, out, 512)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_score_when_burn_ins_cannot_converge(tre, dtype):
    """Smoothing that the chunk burn-ins cannot settle -- alpha 1e-4 (a capped
    burn-in far shorter than 28/alpha), per-model alphas, a model idle for a
    long stretch (burn-ins that see only idle windows) -- is repaired in
    order to the exact sequential values; the repairs are counted."""
    rng = np.random.default_rng(77)
    K, M, win = 40000, 4, 100
    cnt = _score_inputs(rng, K, M)
    for k in cnt:
        cnt[k][20000:30000, 3] = 0                # model 3 idle for a quarter of the series
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = {"w_p": rng.uniform(0.1, 0.3, M), "w_q": rng.uniform(1.0, 3.0, M),
            "alpha": np.array([1e-4, 0.02, 0.5, 0.003]), "theta": rng.uniform(5, 50, M),
            "tau_crit": np.full(M, 0.8), "tau_surplus": np.full(M, 1.2)}
    S, Z, cls, recv = oracle.score(cnt["P"], cnt["D"], cnt["A"], cnt["W"], prof, win, npdt)
    diag = tre.new_diag()
    out = tre.tss_score(_cuda(cnt), prof, win, dtype=dtype, diag=diag)
    np.testing.assert_array_equal(_np(out["S"]), S)
    np.testing.assert_array_equal(_np(out["Z"]), Z)
    np.testing.assert_array_equal(_np(out["cls"]), cls)
    np.testing.assert_array_equal(_np(out["recv"]), recv)
    assert tre.read_diag(diag)["ema_resolved"] > 0


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_score_long_table_idle_stretches(tre, dtype):
    """A table long enough for the burn-ins that skip wholly idle chunks (at
    least 2^22 cells) and for chunks longer than 256 windows (150,000 windows x
    64 models: chunks of 320): models idle for stretches of 3,000 to 20,000
    windows, a sparse model, one that never runs, per-model alphas down to
    0.003, the series split in two calls with the carry between them -- bit
    for bit the sequential values."""
    import torch
    rng = np.random.default_rng(2024)
    K, M, win = 150000, 64, 100
    cnt = _score_inputs(rng, K, M, idle_frac=0.02)
    for m in range(0, M, 5):
        a = int(rng.integers(0, K - 20000))
        cnt_len = int(rng.integers(3000, 20000))
        for k in cnt:
            cnt[k][a:a + cnt_len, m] = 0
    sparse = rng.random(K) < 0.7
    for k in cnt:
        cnt[k][sparse, 7] = 0
        cnt[k][:, 9] = 0
    npdt = np.float32 if dtype == "f32" else np.float64
    alpha = rng.choice(np.array([0.02, 0.05, 0.003, 0.2]), M)
    prof = {"w_p": rng.uniform(0.1, 0.3, M), "w_q": rng.uniform(1.0, 3.0, M),
            "alpha": alpha, "theta": rng.uniform(5, 50, M),
            "tau_crit": np.full(M, 0.8), "tau_surplus": np.full(M, 1.2)}
    S, Z, cls, recv = oracle.score(cnt["P"], cnt["D"], cnt["A"], cnt["W"], prof, win, npdt)
    diag = tre.new_diag()
    out = tre.tss_score(_cuda(cnt), prof, win, dtype=dtype, diag=diag)
    np.testing.assert_array_equal(_np(out["S"]), S)
    np.testing.assert_array_equal(_np(out["Z"]), Z)
    np.testing.assert_array_equal(_np(out["cls"]), cls)
    np.testing.assert_array_equal(_np(out["recv"]), recv)
    assert tre.read_diag(diag)["err"] == 0
    tdt = torch.float32 if dtype == "f32" else torch.float64
    carry = {"S": torch.zeros(M, dtype=tdt, device="cuda"),
             "init": torch.zeros(M, dtype=torch.uint8, device="cuda")}
    parts = []
    for a, b in ((0, 140000), (140000, K)):
        sub = _cuda({k: np.ascontiguousarray(v[a:b]) for k, v in cnt.items()})
        parts.append(tre.tss_score(sub, prof, win, dtype=dtype, carry=carry))
    np.testing.assert_array_equal(np.concatenate([_np(p["S"]) for p in parts]), S)
    np.testing.assert_array_equal(np.concatenate([_np(p["cls"]) for p in parts]), cls)


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("hetero", 0.005)])
def test_calibrate_series_then_normalize(tre, dtype, name, scale):
    """tss_calibrate's smoothed series and idle classes, turned into Z, regions
    and receivers by tss_normalize (in place on the classes), equal the
    oracle's S, Z, cls and recv -- the path the pipeline takes instead of
    smoothing the series a second time."""
    import torch
    w = tracegen.workload(name, scale=scale)
    M, win, K = w["M"], w["window_ms"], w["K"]
    npdt = np.float32 if dtype == "f32" else np.float64
    prof = tracegen.default_profile(M, win)
    o = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], npdt)
    req = _cuda(w["requests"])
    c = tre.tss_window_reduce(M, win, K, requests=req)
    S = torch.empty((K, M), dtype=torch.float32 if dtype == "f32" else torch.float64,
                    device="cuda")
    cls = torch.empty((K, M), dtype=torch.uint8, device="cuda")
    theta = tre.tss_calibrate(c, prof, win, w["slo_ttft_ms"], requests=req, dtype=dtype,
                              S_out=S, cls_out=cls)
    np.testing.assert_array_equal(_np(theta), o["theta"])
    np.testing.assert_array_equal(_np(S), o["S"])
    assert set(np.unique(_np(cls))) <= {oracle.IDLE, oracle.NOM}
    np.testing.assert_array_equal(_np(cls) == oracle.IDLE, o["cls"] == oracle.IDLE)
    out = tre.tss_normalize(S, cls, dict(prof, theta=theta), win, cls_out=cls)
    np.testing.assert_array_equal(_np(out["Z"]), o["Z"])
    np.testing.assert_array_equal(_np(out["cls"]), o["cls"])
    np.testing.assert_array_equal(_np(out["recv"]), o["recv"])
