"""Pins for the oracle's TRE move selection (Sec. IV-B dual-speed control,
Eq. 3, Sec. IV-C bounded pairwise transfer).

* brute force: at every tick, list every admissible (receiver, source) pair
  with a preference key and take the smallest key (a different formulation
  from the oracle's ordered scans), on M <= 4 with unit footprints;
* hand scenarios: idle pool first, floors, pacing cap, heterogeneous
  footprints needing several donor releases;
* invariants on generated traces: budget conservation, floors, no critical
  donor, no idle receiver, rebalance only below the boundary, at most K_p
  transitions per tick, moves only on control ticks.
"""
import numpy as np
import pytest

import oracle
import tracegen

CRIT, NOM, SURP, IDLE = oracle.CRIT, oracle.NOM, oracle.SURP, oracle.IDLE


def _region(z, idle, tc, ts):
    if idle:
        return IDLE
    if z < tc:
        return CRIT
    if z > ts:
        return SURP
    return NOM


def _is_tick(k, win, every):
    return ((k + 1) * win) // every > (k * win) // every


def _brute_walk(Z, cls, tc, ts, win, budget, r0, r_min, fast, slow, Kp):
    """Unit footprints. Returns list of (window, recv, donor, kind, seq) and r."""
    K, M = Z.shape
    r = list(map(int, r0))
    free = budget - sum(r)
    out = []
    for k in range(K):
        f, s = _is_tick(k, win, fast), _is_tick(k, win, slow)
        reg = [_region(Z[k, m], cls[k, m] == IDLE, tc, ts) for m in range(M)]
        mode, recv = 0, None
        if f:
            crit = [(Z[k, m], m) for m in range(M) if reg[m] == CRIT]
            if crit:
                mode, recv = 1, min(crit)[1]
        if mode == 0 and s:
            cands = [(Z[k, m], m) for m in range(M) if reg[m] != IDLE]
            if cands and min(cands)[0] < 1:
                mode, recv = 2, min(cands)[1]
        if mode == 0:
            continue
        for seq in range(Kp):
            sources = []
            if free >= 1:
                sources.append(((0,), -1))
            for d in range(M):
                if d == recv or reg[d] == CRIT or r[d] <= r_min[d]:
                    continue
                if reg[d] == IDLE:
                    sources.append(((1, d), d))
                elif reg[d] == SURP:
                    sources.append(((2, -Z[k, d], d), d))
                elif mode == 1 or Z[k, d] > Z[k, recv]:
                    sources.append(((3, -Z[k, d], d), d))
            if not sources:
                break
            _, d = min(sources)
            if d < 0:
                free -= 1
            else:
                r[d] -= 1
            r[recv] += 1
            out.append((k, recv, d, mode, seq))
    return out, r


def _rand_series(rng, K, M, dtype=np.float64):
    Z = rng.choice(np.array([0.3, 0.5, 0.7, 0.8, 0.9, 1.0, 1.1, 1.2, 1.5, 2.0]), (K, M))
    Z = (Z * rng.choice([1.0, 1.001, 0.999], (K, M))).astype(dtype)
    cls = np.where(rng.random((K, M)) < 0.15, IDLE, NOM).astype(np.uint8)
    return Z, cls


@pytest.mark.parametrize("seed", range(8))
def test_walk_matches_brute_force(seed):
    rng = np.random.default_rng(seed)
    M = 2 + seed % 3
    K = 400
    Z, cls = _rand_series(rng, K, M)
    win = [1000, 500, 2000, 250][seed % 4]
    r0 = rng.integers(1, 4, M)
    budget = int(r0.sum() + seed % 3)
    r_min = rng.integers(0, 2, M).astype(np.int32)
    for Kp in (1, 3):
        for tc in (0.75, 0.95):
            mv, rf, rc = oracle.select_moves(Z, cls, tc, 1.2, win, budget, r0, r_min,
                                             np.ones(M, np.int32), 5000, 10000, Kp)
            ref, rr = _brute_walk(Z, cls, tc, 1.2, win, budget, r0, r_min, 5000, 10000, Kp)
            got = [tuple(int(x) for x in row) for row in mv]
            assert got == ref
            assert rf.tolist() == rr
            assert rc == 0


def _replay_invariants(mv, Z, cls, tc, ts, win, budget, r0, r_min, g, fast, slow, Kp):
    K, M = Z.shape
    r = np.array(r0, np.int64)
    free = budget - int((g * r).sum())
    by_tick = {}
    for k, recv, d, kind, seq in mv:
        by_tick.setdefault(k, []).append((recv, d, kind, seq))
    for k, rows in sorted(by_tick.items()):
        assert _is_tick(k, win, fast) or _is_tick(k, win, slow)
        reg = [_region(Z[k, m], cls[k, m] == IDLE, tc, ts) for m in range(M)]
        seqs = sorted({row[3] for row in rows})
        assert seqs == list(range(len(seqs))) and len(seqs) <= Kp
        for seq in seqs:
            grp = [row for row in rows if row[3] == seq]
            recv, kind = grp[0][0], grp[0][2]
            assert all(row[0] == recv and row[2] == kind for row in grp)
            assert reg[recv] != IDLE
            if kind == oracle.RESCUE:
                assert _is_tick(k, win, fast) and reg[recv] == CRIT
            else:
                assert _is_tick(k, win, slow) and Z[k, recv] < 1
                assert CRIT not in reg or not _is_tick(k, win, fast)
            for _, d, _, _ in grp:
                if d >= 0:
                    assert reg[d] != CRIT and d != recv
                    r[d] -= 1
                    assert r[d] >= r_min[d]
                    free += g[d]
            free -= g[recv]
            r[recv] += 1
            assert free >= 0
            assert int((g * r).sum()) + free == budget
    return r


@pytest.mark.parametrize("name,scale", [("tiny", 1.0), ("mid", 0.02)])
def test_invariants_on_generated_trace(name, scale):
    w = tracegen.workload(name, scale=scale)
    M = w["M"]
    prof = tracegen.default_profile(M, w["window_ms"])
    o = oracle.pipeline_requests(w["requests"], M, w["window_ms"], w["K"], prof,
                                 w["slo_ttft_ms"], np.float64)
    rng = np.random.default_rng(1)
    g = rng.integers(1, 3, M).astype(np.int32)
    budget = int((g * w["r0"]).sum()) + 2
    for Kp in (1, 4):
        for tc in (0.5, 0.8, 0.95):
            mv, rf, rc = oracle.select_moves(o["Z"], o["cls"], tc, 1.2, w["window_ms"], budget,
                                             w["r0"], w["r_min"], g, 5000, 10000, Kp)
            r = _replay_invariants([tuple(int(x) for x in row) for row in mv], o["Z"], o["cls"],
                                   tc, 1.2, w["window_ms"], budget, w["r0"], w["r_min"], g,
                                   5000, 10000, Kp)
            assert r.tolist() == rf.tolist()


def _series(rows):
    Z = np.array([z for z, _ in rows], np.float64)
    cls = np.array([c for _, c in rows], np.uint8)
    return Z, cls


def test_rescue_prefers_idle_pool_then_idle_then_surplus_then_nominal():
    # one window that is a fast and a slow tick (window 9 of 1 s windows ends at 10 s)
    K, M = 10, 5
    Z = np.ones((K, M))
    cls = np.full((K, M), NOM, np.uint8)
    Z[9] = [0.5, 0.6, 1.5, 1.1, 2.0]
    cls[9] = [NOM, NOM, NOM, NOM, IDLE]
    # model 4 idle, model 2 surplus (1.5 > 1.2), model 3 nominal, models 0, 1 critical
    r0 = np.array([1, 1, 2, 2, 2], np.int32)
    g = np.ones(M, np.int32)
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, int(r0.sum()) + 1, r0,
                                    np.ones(M, np.int32), g, 5000, 10000, 8)
    rows = [tuple(int(x) for x in m) for m in mv]
    # window 4 (5 s): fast tick only, Z all 1 -> nothing. Window 9: rescue for model 0
    assert rows == [(9, 0, -1, 1, 0), (9, 0, 4, 1, 1), (9, 0, 2, 1, 2), (9, 0, 3, 1, 3)]
    assert rf.tolist() == [5, 1, 1, 1, 1]


def test_rebalance_nominal_donor_must_be_above_receiver():
    K, M = 10, 3
    Z = np.ones((K, M))
    cls = np.full((K, M), NOM, np.uint8)
    Z[9] = [0.9, 0.95, 0.9]
    r0 = np.array([2, 2, 2], np.int32)
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, 6, r0, np.ones(M, np.int32),
                                    np.ones(M, np.int32), 5000, 10000, 4)
    rows = [tuple(int(x) for x in m) for m in mv]
    # receiver 0 (lowest index among the tie at 0.9); only model 1 (0.95 > 0.9) may donate,
    # once (floor 1)
    assert rows == [(9, 0, 1, 2, 0)]
    assert rf.tolist() == [3, 1, 2]


def test_rescue_blocks_rebalance_even_without_capacity():
    K, M = 10, 2
    Z = np.ones((K, M))
    cls = np.full((K, M), NOM, np.uint8)
    Z[9] = [0.5, 0.7]        # both critical: no donor, no pool
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, 4, np.array([2, 2]),
                                    np.ones(M, np.int32), np.ones(M, np.int32), 5000, 10000, 2)
    assert len(mv) == 0 and rf.tolist() == [2, 2]


def test_heterogeneous_footprints_release_several_donors():
    """A receiver with footprint 2 needs two releases of footprint-1 donors; a
    footprint-2 donor funds a footprint-1 receiver and leaves one unit idle
    (Sec. IV-C: released and activated footprints need not match one for one)."""
    K, M = 10, 3
    Z = np.ones((K, M))
    cls = np.full((K, M), NOM, np.uint8)
    Z[9] = [0.5, 1.5, 1.3]
    g = np.array([2, 1, 1], np.int32)
    r0 = np.array([1, 3, 3], np.int32)
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, 8, r0, np.ones(M, np.int32), g,
                                    5000, 10000, 1)
    rows = [tuple(int(x) for x in m) for m in mv]
    # donors by Z descending among surplus: 1 (1.5) then 1 again (still above floor)
    assert rows == [(9, 0, 1, 1, 0), (9, 0, 1, 1, 0)]
    assert rf.tolist() == [2, 1, 3]
    g = np.array([1, 2, 1], np.int32)
    r0 = np.array([1, 2, 3], np.int32)
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, 8, r0, np.ones(M, np.int32), g,
                                    5000, 10000, 2)
    rows = [tuple(int(x) for x in m) for m in mv]
    # first transition releases model 1 (footprint 2), one unit stays idle;
    # the second uses that idle unit
    assert rows == [(9, 0, 1, 1, 0), (9, 0, -1, 1, 1)]
    assert rf.tolist() == [3, 1, 3]


def test_infeasible_transition_releases_nothing():
    K, M = 10, 2
    Z = np.ones((K, M))
    cls = np.full((K, M), NOM, np.uint8)
    Z[9] = [0.5, 1.5]
    g = np.array([3, 1], np.int32)
    mv, rf, _ = oracle.select_moves(Z, cls, 0.8, 1.2, 1000, 6, np.array([1, 3]),
                                    np.ones(M, np.int32), g, 5000, 10000, 1)
    # the donor can give 2 units (3 -> floor 1), the receiver needs 3
    assert len(mv) == 0 and rf.tolist() == [1, 3]


def test_move_buffer_overflow_reports_required_size():
    rng = np.random.default_rng(2)
    Z, cls = _rand_series(rng, 500, 3)
    full, _, _ = oracle.select_moves(Z, cls, 0.95, 1.2, 1000, 12, np.array([4, 4, 4]),
                                     np.zeros(3, np.int32), np.ones(3, np.int32), 5000, 10000, 2)
    assert len(full) > 3
    lib_moves = np.zeros(3, oracle.MOVE_DTYPE)
    import ctypes as C
    n = np.zeros(1, np.int64)
    r = np.array([4, 4, 4], np.int32)
    rc = oracle.lib().orc_select_f64(
        C.c_int32(3), C.c_int32(1000), C.c_int32(500), oracle._p(Z), oracle._p(cls),
        oracle._p(np.full(3, 0.95)), oracle._p(np.full(3, 1.2)), C.c_int64(12),
        oracle._p(np.zeros(3, np.int32)), oracle._p(np.ones(3, np.int32)), C.c_int32(5000),
        C.c_int32(10000), C.c_int32(2), oracle._p(r), oracle._p(lib_moves), C.c_int64(3),
        oracle._p(n))
    assert rc == 4 and n[0] == len(full)
    np.testing.assert_array_equal(lib_moves, full[:3])


def test_ticks_for_window_lengths():
    # 5 s / 10 s cadences land on the windows whose right edge passes a multiple
    for win, fast, slow in ((100, [49, 99, 149], [99]), (2000, [2, 4, 7, 9], [4, 9]),
                            (3000, [1, 3, 4, 6], [3, 6])):
        ks = range(10 if win >= 2000 else 150)
        assert [k for k in ks if _is_tick(k, win, 5000)][:len(fast)] == fast
        assert [k for k in ks if _is_tick(k, win, 10000)][:len(slow)] == slow
