"""GPU parity of move selection (Sec. IV-B rescue / rebalance, Eq. 3, Sec. IV-C
bounded transfer) on every walk variant of the library, against the oracle's
walk, bit for bit: the warp walk for more than 16 models (shared-memory staged
tick tables and, for long series or many models, tables read from global
memory), the per-tick ranking for 17-32 models and beyond, the thread walk
that visits every tick (cadences that are not nested, or a fast tick shorter
than a window), and pacing caps above 32 on few models."""
import numpy as np
import pytest

import oracle

pytestmark = pytest.mark.gpu

LEVELS = np.array([0.3, 0.5, 0.6, 0.8, 0.8, 0.85, 0.95, 1.0, 1.0, 1.1, 1.2, 1.3, 2.0])


@pytest.fixture(scope="module")
def tre():
    import torch
    import paper_2609_29160_gb300 as lib
    lib.load()
    torch.cuda.set_device(0)
    return lib


def _np(t):
    return t.detach().cpu().numpy()


def _case(seed, K, M, idle=0.1, hetero=False, dtype=np.float32):
    rng = np.random.default_rng(seed)
    Z = rng.choice(LEVELS, (K, M)).astype(dtype)            # many exact ties
    # a few models sit low for long stretches, so rescues repeat on them
    for m in rng.choice(M, max(1, M // 8), replace=False):
        a = int(rng.integers(0, K))
        Z[a: a + K // 5, m] = dtype(0.4)
    cls = np.where(rng.random((K, M)) < idle, oracle.IDLE, oracle.NOM).astype(np.uint8)
    g = rng.integers(1, 4, M).astype(np.int32) if hetero else np.ones(M, np.int32)
    r0 = rng.integers(1, 6, M).astype(np.int32)
    budget = int((g * r0).sum()) + int(rng.integers(0, 4))
    r_min = (rng.random(M) < 0.5).astype(np.int32)
    return Z, cls, g, r0, budget, r_min


def _check(tre, Z, cls, g, r0, budget, r_min, win, cap, fast_ms=5000, slow_ms=10000):
    import torch
    prof = {"w_p": 0.2, "w_q": 2.0, "alpha": 0.2, "theta": 1.0, "tau_crit": 0.8,
            "tau_surplus": 1.2}
    om, orf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, win, budget, r0, r_min, g, fast_ms,
                                     slow_ms, cap)
    Zc, Cc = torch.as_tensor(Z).cuda(), torch.as_tensor(cls).cuda()
    mv, rf, n, diag = tre.tre_select_moves(Zc, Cc, prof, win, budget, r0, r_min, g,
                                           fast_ms=fast_ms, slow_ms=slow_ms, pacing_cap=cap,
                                           moves_cap=len(om) + 8)
    assert n == len(om) and n > 0
    np.testing.assert_array_equal(_np(rf), orf)
    got = np.stack([mv[f].astype(np.int32) for f in ("window", "recv", "donor", "kind", "seq")], 1)
    ref = np.stack([om[f] for f in ("window", "recv", "donor", "kind", "seq")], 1)
    np.testing.assert_array_equal(got, ref)
    assert tre.read_diag(diag)["err"] == 0
    return n


# 17-32 models: one model per lane, per-tick ranking of up to 32 models;
# 33-64: two models per lane; 100: four. K = 3000 one-second windows keeps the
# tick tables in shared memory for up to ~40 models, above that they are read
# from global memory.
@pytest.mark.parametrize("M", [17, 24, 32, 33, 40, 48, 64, 100])
@pytest.mark.parametrize("cap", [1, 3])
def test_warp_walk_many_models(tre, M, cap):
    Z, cls, g, r0, budget, r_min = _case(1000 + M * 7 + cap, 3000, M)
    _check(tre, Z, cls, g, r0, budget, r_min, 1000, cap)


@pytest.mark.parametrize("M", [20, 64])
def test_warp_walk_heterogeneous_footprints(tre, M):
    Z, cls, g, r0, budget, r_min = _case(77 + M, 2000, M, hetero=True)
    _check(tre, Z, cls, g, r0, budget, r_min, 1000, 2)


def test_warp_walk_f64(tre):
    Z, cls, g, r0, budget, r_min = _case(91, 2500, 36, dtype=np.float64)
    _check(tre, Z, cls, g, r0, budget, r_min, 1000, 2)


def test_warp_walk_long_series_sixty_four_models(tre):
    """64 models over 86,400 windows of 100 ms (the streaming workload's model
    count and window length over a tenth of its day): tick tables far beyond
    shared memory."""
    Z, cls, g, r0, budget, r_min = _case(5, 86400, 64, idle=0.05)
    r0 = np.full(64, 8, np.int32)
    budget = 512
    _check(tre, Z, cls, g, r0, budget, r_min, 100, 1)


@pytest.mark.parametrize("M", [6, 12])
@pytest.mark.parametrize("fast_ms,slow_ms,win", [(3000, 10000, 1000), (500, 10000, 1000),
                                                 (700, 2100, 100)])
def test_thread_walk_every_tick(tre, M, fast_ms, slow_ms, win):
    """Cadences that are not nested (slow not a multiple of fast) or a fast
    tick shorter than a window: the walk visits every tick, one thread per
    controller instance."""
    Z, cls, g, r0, budget, r_min = _case(300 + M + fast_ms, 3000, M)
    _check(tre, Z, cls, g, r0, budget, r_min, win, 2, fast_ms, slow_ms)


@pytest.mark.parametrize("M", [5, 16])
def test_pacing_cap_above_thirty_two(tre, M):
    """Few models with a pacing cap of 40 transitions per tick (the sweep's
    caps stop at 8): receivers drain every usable donor in one tick."""
    Z, cls, g, r0, budget, r_min = _case(500 + M, 3000, M)
    r0 = r0 * 12
    budget = int((g * r0).sum())
    _check(tre, Z, cls, g, r0, budget, r_min, 1000, 40)


@pytest.mark.parametrize("caps", [None, list(range(1, 13))])
def test_sweep_twenty_four_models(tre, caps):
    """The sweep's walk launch with more than 16 models: one warp per
    (trace, window length, rescue threshold, pacing cap) instance, eight
    caps to a block (twelve caps: two blocks per (series, threshold))."""
    import tracegen
    sw = tracegen.sweep_workload(scale=0.02, n_traces=1, duration_s=600.0)
    rng = np.random.default_rng(8)
    M0, M = sw["M"], 24
    t = sw["traces"][0]
    t["model"] = (t["model"] + M0 * rng.integers(0, 3, len(t["model"]))).astype(np.int32)
    ext = lambda a: np.resize(np.asarray(a), M)
    sw["M"] = M
    for k in ("w_p", "w_q", "tau_surplus", "slo_ttft_ms", "r0", "r_min", "footprint"):
        if np.ndim(sw[k]):
            sw[k] = ext(sw[k]).astype(np.asarray(sw[k]).dtype)
    sw["budget"] = int(sw["r0"].sum()) + 2
    sw["tau_crit"] = sw["tau_crit"][::3]
    sw["pacing_cap"] = (sw["pacing_cap"][::3] if caps is None
                        else np.asarray(caps, dtype=np.asarray(sw["pacing_cap"]).dtype))
    alpha = [min(1.0, w / 5000.0) for w in sw["window_ms"]]
    import torch
    ref = oracle.sweep(sw["traces"], M, sw["duration_ms"], sw["window_ms"], sw["tau_crit"],
                       sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"], alpha,
                       sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"], sw["footprint"],
                       dtype=np.float32)
    out = tre.tre_sweep([{k: torch.as_tensor(v).cuda() for k, v in t.items()}], M,
                        sw["duration_ms"], sw["window_ms"], alpha, sw["tau_crit"],
                        sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                        sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"], sw["footprint"],
                        moves_cap=512)
    moves = tre.sweep_moves(out, len(ref["instances"]), 512)
    rf = _np(out["r_final"])
    total = 0
    for i, inst in enumerate(ref["instances"]):
        np.testing.assert_array_equal(rf[i], inst["r_final"], err_msg=f"instance {i}")
        om = inst["moves"]
        assert int(_np(out["n_moves"])[i]) == len(om), f"instance {i}"
        got = np.stack([moves[i][f].astype(np.int32)
                        for f in ("window", "recv", "donor", "kind", "seq")], 1) \
            if len(om) else np.zeros((0, 5), np.int32)
        ref_m = np.stack([om[f] for f in ("window", "recv", "donor", "kind", "seq")], 1) \
            if len(om) else np.zeros((0, 5), np.int32)
        np.testing.assert_array_equal(got, ref_m, err_msg=f"instance {i}")
        total += len(om)
    assert total > 0


def test_jump_walk_long_series_sixteen_models(tre):
    """Sixteen models over 43,200 windows of 500 ms (the code/chat workload's
    shape): the jump walk's tables fill nearly all of a block's shared memory,
    and the tick windows are recomputed at each visit instead of staged."""
    Z, cls, g, r0, budget, r_min = _case(16, 43200, 16, idle=0.05)
    for cap in (1, 2):
        _check(tre, Z, cls, g, r0, budget, r_min, 500, cap)


@pytest.mark.parametrize("M", [24, 40])
@pytest.mark.parametrize("fast_ms,slow_ms,win", [(3000, 10000, 1000), (500, 10000, 1000),
                                                 (700, 2100, 100)])
def test_warp_walk_cadences(tre, M, fast_ms, slow_ms, win):
    """The warp walk for more than 16 models on cadences that are not nested
    or a fast tick shorter than a window (every tick visited in order), and on
    nested ones (32 ticks tested against the state at once)."""
    Z, cls, g, r0, budget, r_min = _case(900 + M + fast_ms, 3000, M)
    for cap in (1, 3):
        _check(tre, Z, cls, g, r0, budget, r_min, win, cap, fast_ms, slow_ms)
