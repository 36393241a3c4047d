"""Seeded synthetic request telemetry shaped like the paper's serving workloads.

This module produces INPUTS only: request records (arrival, queue start, first
token, last token, prompt and output lengths) and token-level event streams,
plus the per-model controller settings the workloads are run with. It contains
none of the Token Service Share or TRE arithmetic; both the CPU oracle and the
CUDA library consume what it returns.

The paper evaluates on seven ~720 s serving traces (Sec. VI-A) that are not
available, so these generators stand in for them:

* arrivals are Poisson per model, optionally diurnally modulated and with a
  multiplicative burst window, drawn by Lewis-Shedler thinning;
* prompt/output lengths are rounded log-normals clamped to [1, 131072];
* each model is an FCFS M/M/c queue with c = its initial replica count and
  exponential service time of mean u * cost_m * E[0.2 L_in + L_out];
* a request's service splits into prefill (share 0.2 L_in / (0.2 L_in + L_out))
  and decode (the rest); all times are stored as int32 milliseconds.

Everything is drawn from numpy's PCG64 with an explicit seed, so a workload is
a pure function of its arguments.
"""
from __future__ import annotations

import heapq
import math
from dataclasses import dataclass, field

import numpy as np

MAX_LEN = 131072

# SLO classes (TTFT bound, ms): interactive, best-effort, batch.
SLO_CLASSES_MS = (1000, 5000, 20000)


@dataclass
class TraceSpec:
    n_models: int
    duration_s: float
    n_target: float                      # expected number of requests
    cost: np.ndarray                     # cost weight per model
    share: np.ndarray                    # relative mean arrival rate per model
    len_in: np.ndarray                   # (M, 2) log-normal (mu, sigma) of prompt length
    len_out: np.ndarray                  # (M, 2) log-normal (mu, sigma) of output length
    budget: int                          # replica budget (footprint 1 each)
    r0: np.ndarray | None = None         # initial replicas; None = proportional to load
    rho: float = 0.8                     # utilisation target
    rho_mode: str = "aggregate"          # "aggregate" or "max"
    diurnal_period_s: float = 0.0        # 0 = flat rates
    diurnal_amp: float = 0.0
    burst: tuple | None = None           # (model, start_s, dur_s, factor)
    n_classes: int = 2
    seed: int = 0
    extra: dict = field(default_factory=dict)


def _lognormal_mean(mu, sigma):
    return math.exp(mu + 0.5 * sigma * sigma)


def largest_remainder(weights, total, floor=1):
    """Integer split of `total` proportional to `weights`, each part >= floor."""
    w = np.asarray(weights, dtype=np.float64)
    n = len(w)
    if total < floor * n:
        raise ValueError("budget below the per-model floor")
    ideal = w / w.sum() * total
    base = np.maximum(np.floor(ideal).astype(np.int64), floor)
    while base.sum() > total:                       # floors pushed us over
        i = int(np.argmax(base - ideal))
        base[i] -= 1
    rem = ideal - base
    order = np.lexsort((np.arange(n), -rem))
    i = 0
    while base.sum() < total:
        base[order[i % n]] += 1
        i += 1
    return base.astype(np.int32)


def _rate_fn(spec: TraceSpec, m: int, scale: float):
    base = scale * spec.share[m]
    M = spec.n_models

    def rate(t):
        r = np.full_like(t, base, dtype=np.float64)
        if spec.diurnal_period_s > 0 and spec.diurnal_amp > 0:
            r = r * (1.0 + spec.diurnal_amp *
                     np.sin(2 * np.pi * t / spec.diurnal_period_s + 2 * np.pi * m / M))
        if spec.burst is not None and spec.burst[0] == m:
            _, b0, bd, bf = spec.burst
            r = np.where((t >= b0) & (t < b0 + bd), r * bf, r)
        return r

    peak = base * (1.0 + spec.diurnal_amp)
    if spec.burst is not None and spec.burst[0] == m:
        peak *= spec.burst[3]
    return rate, peak


def _expected_count_unit(spec: TraceSpec):
    grid = np.arange(0.0, spec.duration_s, 0.25) + 0.125
    tot = 0.0
    for m in range(spec.n_models):
        rate, _ = _rate_fn(spec, m, 1.0)
        tot += float(rate(grid).sum()) * 0.25
    return tot


def _fcfs_starts(arr, svc, c):
    """FCFS start times of an M/M/c queue with c identical servers."""
    n = len(arr)
    start = np.empty(n, dtype=np.float64)
    if c <= 0:
        raise ValueError("need at least one server")
    free = [0.0] * c
    heapq.heapify(free)
    a = arr.tolist()
    s = svc.tolist()
    for i in range(n):
        f = free[0]
        st = a[i] if a[i] > f else f
        start[i] = st
        heapq.heapreplace(free, st + s[i])
    return start


def _lengths(rng, mu, sigma, n):
    x = np.rint(rng.lognormal(mu, sigma, size=n))
    return np.clip(x, 1, MAX_LEN).astype(np.int32)


def model_loads(spec: TraceSpec):
    """Mean offered work per second per model (rate * cost * E[0.2 L_in + L_out])."""
    e = np.array([0.2 * _lognormal_mean(*spec.len_in[m]) + _lognormal_mean(*spec.len_out[m])
                  for m in range(spec.n_models)])
    return spec.share * spec.cost * e, e


def initial_replicas(spec: TraceSpec):
    if spec.r0 is not None:
        return np.asarray(spec.r0, dtype=np.int32)
    load, _ = model_loads(spec)
    return largest_remainder(load, spec.budget, floor=1)


def _draw(spec: TraceSpec):
    """Per model: arrival times (s), prompt / output lengths, service times (s)
    and prefill shares, from the spec's seeded generator; plus r0 and u."""
    rng = np.random.Generator(np.random.PCG64(spec.seed))
    M = spec.n_models
    scale = spec.n_target / _expected_count_unit(spec)
    r0 = initial_replicas(spec)
    _, e_work = model_loads(spec)
    lam = scale * spec.share
    # service-time scale u from the utilisation target at base rates
    if spec.rho_mode == "max":
        u = spec.rho / max(lam[m] * spec.cost[m] * e_work[m] / r0[m] for m in range(M))
    else:
        u = spec.rho * r0.sum() / float((lam * spec.cost * e_work).sum())
    draws = []
    for m in range(M):
        rate, peak = _rate_fn(spec, m, scale)
        n_cand = rng.poisson(peak * spec.duration_s)
        t = np.sort(rng.uniform(0.0, spec.duration_s, size=n_cand))
        keep = rng.uniform(0.0, 1.0, size=n_cand) * peak < rate(t)
        t = t[keep]
        n = len(t)
        L_in = _lengths(rng, spec.len_in[m][0], spec.len_in[m][1], n)
        L_out = _lengths(rng, spec.len_out[m][0], spec.len_out[m][1], n)
        svc = rng.exponential(u * spec.cost[m] * e_work[m], size=n)
        pw = 0.2 * L_in
        draws.append((t, L_in, L_out, svc, pw / (pw + L_out)))
    return draws, r0, u


def gen_latent(spec: TraceSpec):
    """Inputs of a closed-loop replay, sorted by arrival: model, arrival (int ms),
    L_in, L_out and the service a request needs once it starts -- whole
    milliseconds to its first token (d_first) and to its last token (d_total;
    equal to d_first when L_out = 1). Same draws as gen_requests."""
    draws, r0, u = _draw(spec)
    cols = {k: [] for k in ("model", "t_arr_ms", "d_first_ms", "d_total_ms", "L_in", "L_out")}
    arr_s = []
    for m, (t, L_in, L_out, svc, f) in enumerate(draws):
        d_total = np.rint(svc * 1000.0).astype(np.int64)
        d_first = np.minimum(np.rint(svc * f * 1000.0).astype(np.int64), d_total)
        d_total = np.where(L_out == 1, d_first, d_total)
        cols["model"].append(np.full(len(t), m, dtype=np.int32))
        cols["t_arr_ms"].append(np.floor(t * 1000.0).astype(np.int64))
        cols["d_first_ms"].append(d_first)
        cols["d_total_ms"].append(d_total)
        cols["L_in"].append(L_in)
        cols["L_out"].append(L_out)
        arr_s.append(t)
    order = np.argsort(np.concatenate(arr_s), kind="stable")
    out = {k: np.ascontiguousarray(np.concatenate(v)[order].astype(np.int32))
           for k, v in cols.items()}
    out["r0"] = r0
    return out


def fcfs_records(lat, M, r):
    """Request records of latent requests served FCFS per model by r[m]
    identical servers, all times in whole milliseconds (the open-loop queue)."""
    n = len(lat["model"])
    start = np.zeros(n, np.int64)
    for m in range(M):
        idx = np.flatnonzero(lat["model"] == m)
        free = [0] * int(r[m])
        heapq.heapify(free)
        for i in idx:
            a = int(lat["t_arr_ms"][i])
            st = max(a, free[0])
            start[i] = st
            heapq.heapreplace(free, st + int(lat["d_total_ms"][i]))
    return {"model": lat["model"].copy(), "t_arr_ms": lat["t_arr_ms"].copy(),
            "t_start_ms": start.astype(np.int32),
            "t_first_ms": (start + lat["d_first_ms"]).astype(np.int32),
            "t_end_ms": (start + lat["d_total_ms"]).astype(np.int32),
            "L_in": lat["L_in"].copy(), "L_out": lat["L_out"].copy()}


def gen_requests(spec: TraceSpec):
    """Request records sorted by arrival. Returns dict of int32 columns + metadata."""
    draws, r0, u = _draw(spec)
    cols = {k: [] for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms",
                            "L_in", "L_out")}
    arr_s = []
    for m, (t, L_in, L_out, svc, f) in enumerate(draws):
        n = len(t)
        start = _fcfs_starts(t, svc, int(r0[m]))
        first = start + svc * f
        end = start + svc
        t_arr = np.floor(t * 1000.0).astype(np.int64)
        t_start = np.floor(start * 1000.0).astype(np.int64)
        t_first = np.floor(first * 1000.0).astype(np.int64)
        t_end = np.floor(end * 1000.0).astype(np.int64)
        t_end = np.where(L_out == 1, t_first, t_end)
        cols["model"].append(np.full(n, m, dtype=np.int32))
        cols["t_arr_ms"].append(t_arr)
        cols["t_start_ms"].append(t_start)
        cols["t_first_ms"].append(t_first)
        cols["t_end_ms"].append(t_end)
        cols["L_in"].append(L_in)
        cols["L_out"].append(L_out)
        arr_s.append(t)
    order = np.argsort(np.concatenate(arr_s), kind="stable")
    out = {}
    for k, v in cols.items():
        a = np.concatenate(v)[order]
        if a.size and (a.max() > np.iinfo(np.int32).max):
            raise ValueError(f"{k} exceeds int32 milliseconds")
        out[k] = np.ascontiguousarray(a.astype(np.int32))
    out["r0"] = r0
    out["u"] = u
    return out


def gen_events(req, seed):
    """Token-level event stream from request records: one record per prompt token
    (spread uniformly over [t_start, t_first]) and one per output token (random
    gaps spanning [t_first, t_end]). Returns SoA columns sorted by (t, req, phase)
    and the per-request table."""
    rng = np.random.Generator(np.random.PCG64(seed))
    n = len(req["model"])
    L_in = req["L_in"].astype(np.int64)
    L_out = req["L_out"].astype(np.int64)
    ts = req["t_start_ms"].astype(np.float64) / 1000.0
    tf = req["t_first_ms"].astype(np.float64) / 1000.0
    te = req["t_end_ms"].astype(np.float64) / 1000.0
    rid = np.arange(n, dtype=np.int32)
    # prefill tokens
    pre_req = np.repeat(rid, L_in)
    u = rng.uniform(0.0, 1.0, size=pre_req.size)
    t_pre = ts[pre_req] + u * (tf - ts)[pre_req]
    # decode tokens: normalised cumulative exponential gaps, first at t_first, last at t_end
    dec_req = np.repeat(rid, L_out)
    g = rng.exponential(1.0, size=dec_req.size)
    starts = np.concatenate(([0], np.cumsum(L_out)[:-1]))
    g[starts] = 0.0
    cs = np.cumsum(g)
    cs -= np.repeat(cs[starts], L_out)
    tot = np.repeat(cs[np.cumsum(L_out) - 1], L_out)
    frac = np.where(tot > 0, cs / np.where(tot > 0, tot, 1.0), 0.0)
    t_dec = tf[dec_req] + frac * (te - tf)[dec_req]
    t = np.concatenate((t_pre, t_dec)).astype(np.float32)
    r = np.concatenate((pre_req, dec_req))
    ph = np.concatenate((np.zeros(pre_req.size, np.uint8), np.ones(dec_req.size, np.uint8)))
    order = np.lexsort((ph, r, t))
    r = r[order]
    return {
        "model": np.ascontiguousarray(req["model"][r]),
        "req": np.ascontiguousarray(r.astype(np.int32)),
        "t_s": np.ascontiguousarray(t[order]),
        "phase": np.ascontiguousarray(ph[order]),
        "req_model": req["model"].copy(),
        "req_t_arr_ms": req["t_arr_ms"].copy(),
        "req_ttft_ms": (req["t_first_ms"] - req["t_arr_ms"]).astype(np.int32),
    }


# ---------------------------------------------------------------------------
# The five workloads. `scale` shrinks the request count (and, where stated,
# nothing else), so reduced cases keep the full structure.
# ---------------------------------------------------------------------------

def _same_lengths(M, li=(6.0, 1.0), lo=(5.0, 0.8)):
    return np.tile(np.array(li), (M, 1)), np.tile(np.array(lo), (M, 1))


def spec_tiny(scale=1.0, seed=0):
    """3 models, cost 1/2/10, replicas 4/3/1, ~10k requests over 600 s, 1 s windows."""
    li, lo = _same_lengths(3)
    return TraceSpec(n_models=3, duration_s=600.0, n_target=10000 * scale,
                     cost=np.array([1.0, 2.0, 10.0]), share=np.array([5.0, 3.0, 1.0]),
                     len_in=li, len_out=lo, budget=8, r0=np.array([4, 3, 1]),
                     rho=0.9, rho_mode="max", n_classes=2, seed=seed)


def spec_mid(scale=1.0, seed=2, duration_s=3600.0):
    """8 models, cost 1..20, 1M requests over 1 h, diurnal, 10x burst for 5 min."""
    M = 8
    li, lo = _same_lengths(M)
    brng = np.random.Generator(np.random.PCG64(seed + 7919))
    b_model = seed % M
    b_start = float(brng.uniform(600.0, 2700.0)) * duration_s / 3600.0
    return TraceSpec(n_models=M, duration_s=duration_s, n_target=1_000_000 * scale,
                     cost=20.0 ** (np.arange(M) / (M - 1)), share=1.0 / (np.arange(M) + 1.0),
                     len_in=li, len_out=lo, budget=64, rho=0.8,
                     diurnal_period_s=duration_s, diurnal_amp=0.5,
                     burst=(b_model, b_start, 300.0 * duration_s / 3600.0, 10.0),
                     n_classes=3, seed=seed)


def spec_hetero(scale=1.0, seed=3):
    """16 models: 8 code-like (long prompts, short outputs), 8 chat-like; 10M over 6 h."""
    M = 16
    li = np.array([(8.0, 1.0)] * 8 + [(5.0, 1.0)] * 8)
    lo = np.array([(4.0, 1.0)] * 8 + [(6.0, 0.8)] * 8)
    share = 1.0 / (np.arange(M) % 8 + 1.0)
    return TraceSpec(n_models=M, duration_s=21600.0, n_target=10_000_000 * scale,
                     cost=20.0 ** (np.arange(M) / (M - 1)), share=share,
                     len_in=li, len_out=lo, budget=128, rho=0.8,
                     diurnal_period_s=21600.0, diurnal_amp=0.5, n_classes=3, seed=seed)


def spec_stream(scale=1.0, seed=4, duration_s=86400.0):
    """64 models with Zipf(1) shares over 24 h; ~230k requests -> ~200M token events."""
    M = 64
    li, lo = _same_lengths(M)
    return TraceSpec(n_models=M, duration_s=duration_s, n_target=230_000 * scale,
                     cost=20.0 ** (np.arange(M) / (M - 1)), share=1.0 / (np.arange(M) + 1.0),
                     len_in=li, len_out=lo, budget=512, rho=0.8, n_classes=3, seed=seed)


SWEEP_WINDOWS_MS = (100, 500, 1000, 2000)
SWEEP_TAU_CRIT = (0.5, 0.6, 0.7, 0.75, 0.8, 0.85, 0.9, 0.95)
SWEEP_PACING = (1, 2, 3, 4, 5, 6, 7, 8)


def default_profile(M, window_ms, dtype=np.float64):
    """Controller profile used by the workloads: w_p=0.2, w_q=2, alpha=min(1, window/5 s),
    tau_crit=0.8, tau_surplus=1.2 (theta comes from calibration)."""
    alpha = min(1.0, window_ms / 5000.0)
    return {
        "w_p": np.full(M, 0.2, dtype), "w_q": np.full(M, 2.0, dtype),
        "alpha": np.full(M, alpha, dtype), "theta": np.ones(M, dtype),
        "tau_crit": np.full(M, 0.8, dtype), "tau_surplus": np.full(M, 1.2, dtype),
    }


def slo_ttft_ms(M, n_classes):
    return np.array([SLO_CLASSES_MS[m % n_classes] for m in range(M)], dtype=np.int32)


def workload(name, scale=1.0, seed=None):
    """One named workload: dict with the request records (or events), grid and controller."""
    if name == "tiny":
        spec, win, dtype = spec_tiny(scale, 0 if seed is None else seed), 1000, "f64"
    elif name == "mid":
        spec, win, dtype = spec_mid(scale, 2 if seed is None else seed), 1000, "f32"
    elif name == "hetero":
        spec, win, dtype = spec_hetero(scale, 3 if seed is None else seed), 500, "f32"
    elif name == "stream":
        spec, win, dtype = spec_stream(scale, 4 if seed is None else seed), 100, "f32"
    else:
        raise ValueError(name)
    req = gen_requests(spec)
    M = spec.n_models
    K = int(round(spec.duration_s * 1000)) // win
    w = {"name": name, "spec": spec, "M": M, "window_ms": win, "K": K, "dtype": dtype,
         "requests": {k: req[k] for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms",
                                          "t_end_ms", "L_in", "L_out")},
         "r0": req["r0"], "budget": int(spec.budget),
         "r_min": np.ones(M, np.int32), "footprint": np.ones(M, np.int32),
         "slo_ttft_ms": slo_ttft_ms(M, spec.n_classes),
         "fast_ms": 5000, "slow_ms": 10000, "pacing_cap": 1}
    if name == "stream":
        w["events"] = gen_events(req, spec.seed + 1)
    return w


def sweep_workload(scale=1.0, n_traces=7, seed0=100, duration_s=3600.0):
    """Open-loop sweep: n_traces mid-like traces (seeds seed0..) x window lengths
    x rescue thresholds x pacing caps."""
    traces = [gen_requests(spec_mid(scale, seed0 + i, duration_s)) for i in range(n_traces)]
    M = 8
    spec = spec_mid(scale, seed0, duration_s)
    return {"name": "sweep", "M": M, "duration_ms": int(round(duration_s * 1000)),
            "traces": [{k: t[k] for k in ("model", "t_arr_ms", "t_start_ms", "t_first_ms",
                                          "t_end_ms", "L_in", "L_out")} for t in traces],
            "r0": traces[0]["r0"], "budget": int(spec.budget),
            "r_min": np.ones(M, np.int32), "footprint": np.ones(M, np.int32),
            "slo_ttft_ms": slo_ttft_ms(M, 3), "window_ms": np.array(SWEEP_WINDOWS_MS, np.int32),
            "tau_crit": np.array(SWEEP_TAU_CRIT), "pacing_cap": np.array(SWEEP_PACING, np.int32),
            "fast_ms": 5000, "slow_ms": 10000,
            "w_p": 0.2, "w_q": 2.0, "tau_surplus": 1.2}
