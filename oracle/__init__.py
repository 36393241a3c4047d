"""CPU oracle for the TSS / TRE hot path (ctypes wrapper around tre_oracle.cpp).

TEST INFRASTRUCTURE ONLY: the slow, plain reference the CUDA library is
checked against. Only tests/, __graft_entry__.smoke() and the CPU-baseline
leg of bench.py may import this package. It shares no code with the library.

Functions take and return numpy arrays laid out [window][model] (row-major).
Pins: every function here is checked in tests/test_oracle_*.py against values
the paper prints (Sec. II-B, Fig. 1 pair), hand-derived traces, closed forms,
brute force on tiny inputs and invariants; see those files for which pin
covers which step.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tre_oracle.cpp")
_OUT = os.path.join(_HERE, "_build", "liboracle.so")

CRIT, NOM, SURP, IDLE = 0, 1, 2, 3
RESCUE, REBALANCE = 1, 2

MOVE_DTYPE = np.dtype([("window", np.int32), ("recv", np.int32), ("donor", np.int32),
                       ("kind", np.int32), ("seq", np.int32)])


def build(force: bool = False) -> str:
    """Compile the oracle with plain IEEE arithmetic (no contraction, no fast-math)."""
    if force or not os.path.exists(_OUT) or os.path.getmtime(_OUT) < os.path.getmtime(_SRC):
        os.makedirs(os.path.dirname(_OUT), exist_ok=True)
        tmp = _OUT + f".tmp{os.getpid()}"
        subprocess.run(["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math",
                        "-fPIC", "-shared", _SRC, "-o", tmp], check=True)
        os.replace(tmp, _OUT)
    return _OUT


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(build())
        assert _lib.orc_move_size() == MOVE_DTYPE.itemsize
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


def _req_cols(req):
    return [_i32(req[k]) for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms",
                                   "t_end_ms", "L_in", "L_out")]


def reduce_requests(req, M, window_ms, K):
    """Per-window prompt (P) and decode (D) token counts and running (A) /
    waiting (W) gauges from request records. Returns (P, D, A, W, drops[3])."""
    cols = _req_cols(req)
    n = len(cols[0])
    P, D, A, W = (np.zeros((K, M), np.int32) for _ in range(4))
    drops = np.zeros(3, np.int64)
    rc = lib().orc_reduce_requests(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                   C.c_int64(n), *[_p(c) for c in cols],
                                   _p(P), _p(D), _p(A), _p(W), _p(drops))
    if rc:
        raise ValueError("oracle: bad arguments")
    return P, D, A, W, drops


def occupancy_mean_requests(req, M, window_ms, K):
    """Per-window request-milliseconds running (A_ms) and waiting (W_ms) inside
    each window (time-averaged occupancy = these / window_ms). int64 [K, M]."""
    cols = _req_cols(req)
    A_ms, W_ms = np.zeros((K, M), np.int64), np.zeros((K, M), np.int64)
    rc = lib().orc_occupancy_mean_requests(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                           C.c_int64(len(cols[0])), *[_p(c) for c in cols],
                                           _p(A_ms), _p(W_ms))
    if rc:
        raise ValueError("oracle: bad arguments")
    return A_ms, W_ms


def class_models(model, cls, M, n_classes):
    """Model ids of (model, SLO class) pairs: model * n_classes + class, -1 if
    either is out of range."""
    model, cls = _i32(model), _i32(cls)
    out = np.zeros(len(model), np.int32)
    rc = lib().orc_class_models(C.c_int64(len(model)), _p(model), _p(cls), C.c_int32(M),
                                C.c_int32(n_classes), _p(out))
    if rc:
        raise ValueError("oracle: bad arguments")
    return out


def slo_counts_requests(req, M, window_ms, K, slo_ttft_ms):
    cols = _req_cols(req)
    n_arr, n_met = np.zeros((K, M), np.int32), np.zeros((K, M), np.int32)
    rc = lib().orc_slo_counts_requests(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                       C.c_int64(len(cols[0])), *[_p(c) for c in cols],
                                       _p(_i32(slo_ttft_ms)), _p(n_arr), _p(n_met))
    if rc:
        raise ValueError("oracle: bad arguments")
    return n_arr, n_met


def reduce_events(ev, M, window_ms, K):
    model, req = _i32(ev["model"]), _i32(ev["req"])
    t_s = np.ascontiguousarray(ev["t_s"], dtype=np.float32)
    phase = np.ascontiguousarray(ev["phase"], dtype=np.uint8)
    rm, rta = _i32(ev["req_model"]), _i32(ev["req_t_arr_ms"])
    P, D, A, W = (np.zeros((K, M), np.int32) for _ in range(4))
    drops = np.zeros(3, np.int64)
    rc = lib().orc_reduce_events(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                 C.c_int64(len(model)), _p(model), _p(req), _p(t_s), _p(phase),
                                 C.c_int64(len(rm)), _p(rm), _p(rta),
                                 _p(P), _p(D), _p(A), _p(W), _p(drops))
    if rc:
        raise ValueError("oracle: bad arguments")
    return P, D, A, W, drops


def occupancy_mean_events(ev, M, window_ms, K):
    """Time-averaged occupancy of token events: request-milliseconds running
    (first to last valid event) and waiting (arrival to first event) per window.
    int64 [K, M]."""
    model, req = _i32(ev["model"]), _i32(ev["req"])
    t_s = np.ascontiguousarray(ev["t_s"], dtype=np.float32)
    phase = np.ascontiguousarray(ev["phase"], dtype=np.uint8)
    rm, rta = _i32(ev["req_model"]), _i32(ev["req_t_arr_ms"])
    A_ms, W_ms = np.zeros((K, M), np.int64), np.zeros((K, M), np.int64)
    rc = lib().orc_occupancy_mean_events(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                         C.c_int64(len(model)), _p(model), _p(req), _p(t_s),
                                         _p(phase), C.c_int64(len(rm)), _p(rm), _p(rta),
                                         _p(A_ms), _p(W_ms))
    if rc:
        raise ValueError("oracle: bad arguments")
    return A_ms, W_ms


def slo_counts_events(ev, M, window_ms, K, slo_ttft_ms):
    rm, rta, rtt = _i32(ev["req_model"]), _i32(ev["req_t_arr_ms"]), _i32(ev["req_ttft_ms"])
    n_arr, n_met = np.zeros((K, M), np.int32), np.zeros((K, M), np.int32)
    rc = lib().orc_slo_counts_events(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                     C.c_int64(len(rm)), _p(rm), _p(rta), _p(rtt),
                                     _p(_i32(slo_ttft_ms)), _p(n_arr), _p(n_met))
    if rc:
        raise ValueError("oracle: bad arguments")
    return n_arr, n_met


def _suffix(dtype):
    dtype = np.dtype(dtype)
    if dtype == np.float32:
        return "f32"
    if dtype == np.float64:
        return "f64"
    raise ValueError(dtype)


def _prof(profile, M, dtype):
    return {k: np.ascontiguousarray(np.broadcast_to(np.asarray(profile[k], dtype=dtype), (M,)))
            for k in ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")}


def score(P, D, A, W, profile, window_ms, dtype=np.float64, carry=None, occ_ms=None):
    """Eq. 1 raw TSS -> EMA -> Eq. 2 Z -> region. Returns (S, Z, cls, recv).
    carry: optional dict {"S": [M], "init": [M] uint8} updated in place.
    occ_ms: optional (A_ms, W_ms) int64 -- time-averaged occupancy instead of
    the sampled A, W."""
    K, M = P.shape
    pr = _prof(profile, M, dtype)
    S = np.zeros((K, M), dtype)
    Z = np.zeros((K, M), dtype)
    cls = np.zeros((K, M), np.uint8)
    recv = np.zeros(K, np.int32)
    f = getattr(lib(), "orc_score_" + _suffix(dtype))
    rc = f(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
           *[_p(_i32(a)) for a in (P, D, A, W)],
           *[_p(pr[k]) for k in ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")],
           _p(carry["S"]) if carry else None, _p(carry["init"]) if carry else None,
           _p(S), _p(Z), _p(cls), _p(recv),
           *((_p(np.ascontiguousarray(occ_ms[0], np.int64)),
              _p(np.ascontiguousarray(occ_ms[1], np.int64))) if occ_ms is not None
             else (None, None)))
    if rc:
        raise ValueError("oracle: bad arguments")
    return S, Z, cls, recv


def rank(Z, cls):
    """Per window the Eq. 3 receiver (-1 if all idle) and its first 8 donors in
    acquisition order (Sec. IV-B), -1 in unused slots. Returns (recv, order)."""
    K, M = Z.shape
    recv = np.zeros(K, np.int32)
    order = np.zeros((K, 8), np.int32)
    f = getattr(lib(), "orc_rank_" + _suffix(Z.dtype))
    rc = f(C.c_int32(M), C.c_int32(K), _p(np.ascontiguousarray(Z)),
           _p(np.ascontiguousarray(cls, np.uint8)), _p(recv), _p(order))
    if rc:
        raise ValueError("oracle: bad arguments")
    return recv, order


def calibrate(S, cls, n_arr, n_met, ok_frac=0.95, reliability=0.95):
    """theta per model (Sec. III-B). Returns (theta[M], n_degenerate)."""
    K, M = S.shape
    theta = np.zeros(M, S.dtype)
    deg = np.zeros(1, np.int64)
    f = getattr(lib(), "orc_calibrate_" + _suffix(S.dtype))
    rc = f(C.c_int32(M), C.c_int32(K), _p(np.ascontiguousarray(S)),
           _p(np.ascontiguousarray(cls, np.uint8)), _p(_i32(n_arr)), _p(_i32(n_met)),
           C.c_double(ok_frac), C.c_double(reliability), _p(theta), _p(deg))
    if rc:
        raise ValueError("oracle: bad arguments")
    return theta, int(deg[0])


def select_moves(Z, cls, tau_crit, tau_surplus, window_ms, budget, r0, r_min, footprint,
                 fast_ms=5000, slow_ms=10000, pacing_cap=1, cap=None):
    """Open-loop TRE move selection. Returns (moves structured array, r_final, status)."""
    K, M = Z.shape
    dtype = Z.dtype
    tc = np.ascontiguousarray(np.broadcast_to(np.asarray(tau_crit, dtype), (M,)))
    ts = np.ascontiguousarray(np.broadcast_to(np.asarray(tau_surplus, dtype), (M,)))
    r = _i32(r0).copy()
    if cap is None:
        cap = 1024
    while True:
        moves = np.zeros(cap, MOVE_DTYPE)
        n = np.zeros(1, np.int64)
        rr = r.copy()
        f = getattr(lib(), "orc_select_" + _suffix(dtype))
        rc = f(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K), _p(np.ascontiguousarray(Z)),
               _p(np.ascontiguousarray(cls, np.uint8)), _p(tc), _p(ts), C.c_int64(budget),
               _p(_i32(r_min)), _p(_i32(footprint)), C.c_int32(fast_ms), C.c_int32(slow_ms),
               C.c_int32(pacing_cap), _p(rr), _p(moves), C.c_int64(cap), _p(n))
        if rc == 1:
            raise ValueError("oracle: bad arguments")
        if rc == 4:
            cap = int(n[0])
            continue
        return moves[: int(n[0])], rr, rc


def closed_loop(lat, M, window_ms, K, profile, budget, r0, r_min, footprint, tau_crit,
                tau_surplus, fast_ms=5000, slow_ms=10000, pacing_cap=1, dtype=np.float64,
                cap=None, wake_ms=0, sleep_ms=0, guard_ms=None):
    """Closed-loop replay of latent requests (model, t_arr_ms, d_first_ms,
    d_total_ms, L_in, L_out): the controller's moves change the servers, the
    served requests make the telemetry it scores. profile holds w_p, w_q,
    alpha, theta. wake_ms / sleep_ms: actuation delays of a receiver replica
    and of a released donor replica (after it drains). guard_ms: per-model
    latency guard (a first token later than this after arrival breaches it),
    None = no guard. Returns dict with the served records (t_start_ms,
    t_first_ms, t_end_ms), moves, r_final, Z, cls."""
    n = len(lat["model"])
    pr = _prof(dict(profile, tau_crit=tau_crit, tau_surplus=tau_surplus), M, dtype)
    out = {k: np.zeros(n, np.int32) for k in ("t_start_ms", "t_first_ms", "t_end_ms")}
    Z = np.zeros((K, M), dtype)
    cls = np.zeros((K, M), np.uint8)
    r = np.zeros(M, np.int32)
    cap = 1 << 16 if cap is None else cap
    while True:
        moves = np.zeros(cap, MOVE_DTYPE)
        nm = np.zeros(1, np.int64)
        f = getattr(lib(), "orc_closed_loop_" + _suffix(dtype))
        rc = f(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K), C.c_int64(n),
               *[_p(_i32(lat[k])) for k in ("model", "t_arr_ms", "d_first_ms", "d_total_ms",
                                            "L_in", "L_out")],
               *[_p(pr[k]) for k in ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")],
               C.c_int64(budget), _p(_i32(r0)), _p(_i32(r_min)), _p(_i32(footprint)),
               C.c_int32(fast_ms), C.c_int32(slow_ms), C.c_int32(pacing_cap),
               C.c_int32(wake_ms), C.c_int32(sleep_ms),
               _p(_i32(guard_ms)) if guard_ms is not None else None,
               _p(out["t_start_ms"]), _p(out["t_first_ms"]), _p(out["t_end_ms"]), _p(r),
               _p(moves), C.c_int64(cap), _p(nm), _p(Z), _p(cls))
        if rc == 1:
            raise ValueError("oracle: bad arguments")
        if rc == 4:
            cap = int(nm[0])
            continue
        break
    rec = {"model": _i32(lat["model"]), "t_arr_ms": _i32(lat["t_arr_ms"]), **out,
           "L_in": _i32(lat["L_in"]), "L_out": _i32(lat["L_out"])}
    return {"records": rec, "moves": moves[: int(nm[0])], "r_final": r, "Z": Z, "cls": cls}


def slo_tpot_counts_requests(req, M, window_ms, K, tpot_ms):
    """Per (arrival window, model): requests with L_out > 1 and how many met
    (t_end - t_first) <= tpot_ms * (L_out - 1)."""
    cols = _req_cols(req)
    n_dec, n_met = np.zeros((K, M), np.int32), np.zeros((K, M), np.int32)
    rc = lib().orc_slo_tpot_counts_requests(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                            C.c_int64(len(cols[0])), *[_p(c) for c in cols],
                                            _p(_i32(tpot_ms)), _p(n_dec), _p(n_met))
    if rc:
        raise ValueError("oracle: bad arguments")
    return n_dec, n_met


def stage_gauges(req, M, window_ms, K):
    """Running requests split at the first token, read at each window's last
    millisecond: in prefill on [t_start, t_first) and decoding on
    [t_first, t_end), among the records reduce_requests keeps. Returns
    (A_prefill, A_decode)."""
    cols = _req_cols(req)
    A_p, A_d = np.zeros((K, M), np.int32), np.zeros((K, M), np.int32)
    rc = lib().orc_stage_gauges_requests(C.c_int32(M), C.c_int32(window_ms), C.c_int32(K),
                                         C.c_int64(len(cols[0])), *[_p(c) for c in cols],
                                         _p(A_p), _p(A_d))
    if rc:
        raise ValueError("oracle: bad arguments")
    return A_p, A_d


def stage_pipeline(req, M, window_ms, K, profile, slo_ttft_ms, slo_tpot_ms, dtype,
                   ok_frac=0.95, reliability=0.95):
    """Stage-aware signal (separate prefill and decode states, Sec. VIII):
    prefill TSS = (P/dt) / max(A_prefill + w_q*W, 1), calibrated on TTFT;
    decode TSS = (D/dt) / max(A_decode, 1), calibrated on TPOT. Each stage is
    smoothed, calibrated and normalised like the scalar signal."""
    P, D, A, W, drops = reduce_requests(req, M, window_ms, K)
    A_p, A_d = stage_gauges(req, M, window_ms, K)
    zero = np.zeros_like(P)
    n_arr, n_met = slo_counts_requests(req, M, window_ms, K, slo_ttft_ms)
    n_dec, n_met_d = slo_tpot_counts_requests(req, M, window_ms, K, slo_tpot_ms)
    out = {"A_prefill": A_p, "A_decode": A_d}
    for stage, cnt, counts in (("prefill", (P, zero, A_p, W), (n_arr, n_met)),
                               ("decode", (zero, D, A_d, zero), (n_dec, n_met_d))):
        prof = dict(profile, w_p=1.0) if stage == "prefill" else dict(profile)
        S, _, cls, _ = score(*cnt, prof, window_ms, dtype)
        theta, deg = calibrate(S, cls, *counts, ok_frac, reliability)
        S, Z, cls, _ = score(*cnt, dict(prof, theta=theta), window_ms, dtype)
        out[stage] = {"S": S, "Z": Z, "cls": cls, "theta": theta, "degenerate": deg}
    return out


def pipeline_requests(req, M, window_ms, K, profile, slo_ttft_ms, dtype, ok_frac=0.95,
                      reliability=0.95, mean_occupancy=False):
    """Reduce -> score (S) -> calibrate theta -> score (Z, class, receiver).
    mean_occupancy: Eq. 1's running and waiting counts as window means."""
    P, D, A, W, drops = reduce_requests(req, M, window_ms, K)
    occ = occupancy_mean_requests(req, M, window_ms, K) if mean_occupancy else None
    n_arr, n_met = slo_counts_requests(req, M, window_ms, K, slo_ttft_ms)
    S, _, cls, _ = score(P, D, A, W, profile, window_ms, dtype, occ_ms=occ)
    theta, deg = calibrate(S, cls, n_arr, n_met, ok_frac, reliability)
    prof = dict(profile)
    prof["theta"] = theta
    S, Z, cls, recv = score(P, D, A, W, prof, window_ms, dtype, occ_ms=occ)
    out = {"P": P, "D": D, "A": A, "W": W, "drops": drops, "n_arr": n_arr, "n_met": n_met,
           "S": S, "Z": Z, "cls": cls, "recv": recv, "theta": theta, "degenerate": deg}
    if occ is not None:
        out["A_ms"], out["W_ms"] = occ
    return out


def sweep(traces, M, duration_ms, window_ms_list, tau_crit_list, pacing_list, w_p, w_q,
          tau_surplus, alpha_list, slo_ttft_ms, budget, r0, r_min, footprint, fast_ms=5000,
          slow_ms=10000, dtype=np.float32, ok_frac=0.95, reliability=0.95, series_hook=None):
    """Open-loop sweep: for every trace and window length, reduce the records at
    that window length directly, calibrate theta, score; then run the move
    selection for every (rescue threshold, pacing cap) setting."""
    out = {"series": [], "instances": []}
    for ti, req in enumerate(traces):
        for wi, win in enumerate(window_ms_list):
            K = duration_ms // int(win)
            prof = {"w_p": w_p, "w_q": w_q, "alpha": alpha_list[wi], "theta": 1.0,
                    "tau_crit": tau_crit_list[0], "tau_surplus": tau_surplus}
            s = pipeline_requests(req, M, int(win), K, prof, slo_ttft_ms, dtype, ok_frac,
                                  reliability)
            s["trace"], s["window_ms"], s["K"] = ti, int(win), K
            out["series"].append(s if series_hook is None else series_hook(s))
            for tau in tau_crit_list:
                for cap in pacing_list:
                    mv, rf, _ = select_moves(s["Z"], s["cls"], tau, tau_surplus, int(win), budget,
                                             r0, r_min, footprint, fast_ms, slow_ms, int(cap))
                    out["instances"].append({"moves": mv, "r_final": rf})
    return out
