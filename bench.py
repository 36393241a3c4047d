#!/usr/bin/env python
"""Benchmark: the open-loop TSS + TRE sweep on one batch of synthetic telemetry.

A step is one tre_sweep call: 7 synthetic one-hour traces of ~1M request
records each (8 models, diurnal load, a 10x burst), reduced at 100 ms and
aggregated exactly to 0.5 / 1 / 2 s windows, theta calibrated for each of the
28 (trace, window) series, scored, and the TRE controller run for all 256
settings (4 window lengths x 8 rescue thresholds x 8 pacing caps) -- 1792
controller instances. Inputs stay resident in HBM for the device-timed value;
the e2e number copies the records in from pinned host memory and the results
out every step.

Prints one JSON line (rank 0). `--impl reference` times the CPU oracle on a
bounded sample of the same workload instead.
"""
import argparse
import ctypes as C
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import tracegen  # noqa: E402

METRIC = "telemetry events/sec and model-windows/sec through TSS+selection; % of HBM peak"
UNIT = "events/s"
WORKLOAD = "sweep: 7 traces x 1M requests (8 models, 1 h), 4 window lengths x 8 rescue thresholds x 8 pacing caps"


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--scale", type=float, default=1.0, help="request-count scale (1.0 = full)")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-graph", action="store_true",
                    help="issue the timed calls one by one instead of as one CUDA graph")
    ap.add_argument("--no-replay", action="store_true",
                    help="skip the closed-loop replay measured beside the sweep")
    ap.add_argument("--no-configs", action="store_true",
                    help="skip the single-trace workloads measured beside the sweep")
    return ap.parse_args()


def host_mapped(ptr):
    """True when the GPU addresses the pinned host allocation at `ptr` under
    the same address (unified addressing), asked of the CUDA runtime."""
    try:
        rt = C.CDLL("libcudart.so")
    except OSError:
        try:
            import glob
            cands = sorted(glob.glob(os.path.join(os.environ.get("CUDA_HOME", "/usr/local/cuda"),
                                                  "lib64", "libcudart.so*")))
            rt = C.CDLL(cands[-1])
        except (OSError, IndexError):
            return False
    dptr = C.c_void_p()
    rc = rt.cudaHostGetDevicePointer(C.byref(dptr), C.c_void_p(ptr), C.c_uint(0))
    return rc == 0 and dptr.value == ptr


SWEEP_SEED0 = 100          # the sweep's traces are seeded 100 .. 106


def idle_rank(dist, world, dev="cuda"):
    """A rank with no trace of the sweep (more ranks than traces): it joins the
    barriers and the whole-job reductions with nothing of its own."""
    dist.barrier()
    dist.barrier()
    over_ranks(dist, dev, 0.0, [0, 0, 0, 0, 0])
    over_ranks(dist, dev, 0.0, [])
    dist.destroy_process_group()


def over_ranks(dist, device, ms, units):
    """Whole-job figures of a multi-rank run: the slowest rank's milliseconds
    and the units (records, model-windows) summed over all ranks."""
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    if not units:
        return float(t.item()), []
    u = torch.tensor([float(x) for x in units], dtype=torch.float64, device=device)
    dist.all_reduce(u, op=dist.ReduceOp.SUM)
    return float(t.item()), [float(x) for x in u.tolist()]


def alphas(windows):
    return [min(1.0, w / 5000.0) for w in windows]


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi clocks / throttle reasons, sampled every 100 ms while the
    sampler runs; window() keeps the samples taken between two marks (host wall
    time, compared with nvidia-smi's own timestamps)."""
    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu):
        self.gpu = gpu
        self.proc = None
        self.rows = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    @staticmethod
    def now():
        import datetime
        return datetime.datetime.now()

    def stop(self):
        if self.proc is None:
            return
        time.sleep(0.15)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out = ""
        import datetime
        for r in out.strip().splitlines():
            f = [x.strip() for x in r.split(",")]
            if len(f) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f")
                sm, mx = float(f[2]), float(f[3])
            except ValueError:
                continue
            self.rows.append((ts, sm, mx, [n for i, n in enumerate(self.NAMES)
                                           if f[6 + i].lower() == "active"]))

    def window(self, t0, t1, what):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"],
                    "samples": 0, "window": what}
        rows = [r for r in self.rows if t0 <= r[0] <= t1]
        reasons = sorted({n for r in rows for n in r[3]})
        return {"sm_mhz": statistics.median([r[1] for r in rows]) if rows else None,
                "sm_max_mhz": max(r[2] for r in rows) if rows else None,
                "reasons": reasons, "samples": len(rows), "window": what}


def _oracle_sweep(sw):
    import oracle
    oracle.sweep(sw["traces"], sw["M"], sw["duration_ms"], sw["window_ms"], sw["tau_crit"],
                 sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                 alphas(sw["window_ms"]), sw["slo_ttft_ms"], sw["budget"], sw["r0"],
                 sw["r_min"], sw["footprint"], dtype=np.float32)


def run_reference(args):
    """The CPU oracle, as it stands, on a bounded sample of the workload: one
    trace, cut to a duration that keeps the whole --steps/--warmup run near
    90 s (sized from a 60 s probe), with all window lengths and all 64
    controller settings."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    # the same request rate over a shorter trace: scale with the duration
    probe = tracegen.sweep_workload(scale=args.scale * 60.0 / 3600.0, n_traces=1,
                                    duration_s=60.0)
    t0 = time.perf_counter()
    _oracle_sweep(probe)
    rate = len(probe["traces"][0]["model"]) / max(time.perf_counter() - t0, 1e-6)
    per_step = 90.0 / max(1, args.steps + args.warmup)
    rec_per_trace_s = max(len(probe["traces"][0]["model"]) / 60.0, 1e-6)
    dur = per_step * rate / rec_per_trace_s
    dur = float(min(3600, max(10, int(dur // 10) * 10)))   # whole slow ticks
    sw = tracegen.sweep_workload(scale=args.scale * dur / 3600.0, n_traces=1, duration_s=dur)
    n_rec = len(sw["traces"][0]["model"])
    for _ in range(args.warmup):
        _oracle_sweep(sw)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _oracle_sweep(sw)
    dt = time.perf_counter() - t0
    v = n_rec * args.steps / dt
    sample = (f"1 trace cut to {dur:.0f} s ({n_rec} records) of the one-hour workload, "
              f"4 window lengths, 64 settings per step")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
        "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": {"workload": WORKLOAD, "sample": sample},
        "cpu_baseline": {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}))


def host_cpu():
    """The host's CPU model and core count, as lscpu reports them (for the CPU
    baselines)."""
    info = {"nproc": os.cpu_count()}
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            k, _, v = line.partition(":")
            if k.strip() in ("Model name", "Architecture", "Vendor ID"):
                info[k.strip().lower().replace(" ", "_")] = v.strip()
    except Exception:
        pass
    return info


def cpu_baseline(scale):
    import oracle
    sw = tracegen.sweep_workload(scale=scale, n_traces=1)
    n_rec = len(sw["traces"][0]["model"])
    t0 = time.perf_counter()
    oracle.sweep(sw["traces"], sw["M"], sw["duration_ms"], sw["window_ms"], sw["tau_crit"],
                 sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                 alphas(sw["window_ms"]), sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"],
                 sw["footprint"], dtype=np.float32)
    dt = time.perf_counter() - t0
    return {"value": n_rec / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"1 of the 7 traces ({n_rec} records), all 4 window lengths, all 64 settings; {dt:.1f} s"}


# The oracle spread over the host's cores: the sweep's independent (trace,
# window length) units -- each a reduction, calibration and scoring plus its 64
# controller walks -- in worker processes (spawned, never forked after CUDA
# use); each worker generates the seven traces once before the timed map.
_PAR_TRACES = None


def _par_init(scale, seed0):
    global _PAR_TRACES
    sw = tracegen.sweep_workload(scale=scale, seed0=seed0)
    _PAR_TRACES = sw


def _par_unit(unit):
    import oracle
    ti, wi = unit
    sw = _PAR_TRACES
    oracle.sweep([sw["traces"][ti]], sw["M"], sw["duration_ms"], [int(sw["window_ms"][wi])],
                 sw["tau_crit"], sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                 [alphas(sw["window_ms"])[wi]], sw["slo_ttft_ms"], sw["budget"], sw["r0"],
                 sw["r_min"], sw["footprint"], dtype=np.float32)
    return len(sw["traces"][ti]["model"]) if wi == 0 else 0


def cpu_baseline_parallel(scale, seed0):
    """The whole sweep on the oracle, its (trace, window length) units spread
    over one process per host core; wall time of the map only."""
    import multiprocessing as mp
    n_proc = max(1, os.cpu_count() or 1)
    try:
        ctx = mp.get_context("spawn")
        with ctx.Pool(n_proc, initializer=_par_init, initargs=(scale, seed0)) as pool:
            # bounded waits: a worker that dies must not stall the bench
            pool.map_async(_par_unit, [(0, 0)] * n_proc).get(timeout=300)
            units = [(t, w) for t in range(7) for w in range(4)]
            t0 = time.perf_counter()
            n_rec = sum(pool.map_async(_par_unit, units, chunksize=1).get(timeout=300))
            dt = time.perf_counter() - t0
    except Exception as e:   # a baseline must not cost the bench line
        return {"error": f"{type(e).__name__}: {e}"}
    return {"value": n_rec / dt, "unit": UNIT, "cores": n_proc, "kind": "oracle",
            "sample": f"the whole sweep: 7 traces ({n_rec} records) x 4 window lengths x 64 "
                      f"settings as 28 (trace, window length) units over {n_proc} processes; "
                      f"{dt:.1f} s"}


# ---------------------------------------------------------------------------
# The single-trace workloads: one pass of the whole path per step
# (tss_window_reduce -> tss_calibrate -> tss_normalize -> tre_select_moves).
# ---------------------------------------------------------------------------
CONFIGS = (
    # (key, workload name, dtypes, timed steps, oracle sample: fraction of the
    # trace's duration kept, from its start)
    ("tiny_3_models_600s", "tiny", ("f64", "f32"), 50, 1.0),
    ("mid_8_models_1M_requests_1h", "mid", ("f32", "f64"), 30, 1.0),
    ("hetero_16_models_10M_requests_6h", "hetero", ("f32",), 20, 1.0 / 8),
    ("stream_64_models_200M_token_events_24h", "stream", ("f32",), 10, 1.0 / 24),
)


def config_bytes(w, tsize):
    """Algorithmic bytes of one pass: the telemetry read once (28 B per request
    record, or 13 B per token event plus 12 B per request-table row) and, per
    (window, model), the four counts, S and Z in the profile's type and the
    region byte written once."""
    KM = w["K"] * w["M"]
    if "events" in w:
        src = len(w["events"]["model"]) * 13 + len(w["events"]["req_model"]) * 12
    else:
        src = len(w["requests"]["model"]) * 28
    return src + KM * (16 + 2 * tsize + 1)


def cut_workload(w, frac):
    """The first `frac` of a workload's duration: requests arriving (events
    stamped) before the cut, on the windows before it."""
    if frac >= 1.0:
        return w
    K = max(1, int(w["K"] * frac))
    cut = K * w["window_ms"]
    out = dict(w, K=K)
    if "events" in w:
        ev = w["events"]
        keep = ev["t_s"].astype(np.float64) * 1000.0 < cut
        out["events"] = {k: (v[keep] if len(v) == len(keep) and k in ("model", "req", "t_s",
                                                                      "phase") else v)
                         for k, v in ev.items()}
    keep = w["requests"]["t_arr_ms"] < cut
    out["requests"] = {k: v[keep] for k, v in w["requests"].items()}
    return out


def _oracle_path(w, dtype):
    """The oracle's whole path for one trace (reduce, SLO counts, score,
    calibrate, score, walk)."""
    import oracle
    M, win, K = w["M"], w["window_ms"], w["K"]
    prof = tracegen.default_profile(M, win)
    Z, cls = _oracle_models(w, dtype, prof)
    oracle.select_moves(Z, cls, 0.8, 1.2, win, w["budget"], w["r0"], w["r_min"], w["footprint"],
                        w["fast_ms"], w["slow_ms"], w["pacing_cap"])


def _oracle_models(w, dtype, prof):
    import oracle
    M, win, K = w["M"], w["window_ms"], w["K"]
    if "events" in w:
        ev = w["events"]
        P, D, A, W, _ = oracle.reduce_events(ev, M, win, K)
        n_arr, n_met = oracle.slo_counts_events(ev, M, win, K, w["slo_ttft_ms"])
        S, _, cls, _ = oracle.score(P, D, A, W, prof, win, dtype)
        theta, _ = oracle.calibrate(S, cls, n_arr, n_met)
        _, Z, cls, _ = oracle.score(P, D, A, W, dict(prof, theta=theta), win, dtype)
        return Z, cls
    o = oracle.pipeline_requests(w["requests"], M, win, K, prof, w["slo_ttft_ms"], dtype)
    return o["Z"], o["cls"]


def _model_slice(w, m):
    """Model m's telemetry as a one-model workload (ids remapped to 0; token
    events' request ids renumbered within the model)."""
    one = {"M": 1, "window_ms": w["window_ms"], "K": w["K"],
           "slo_ttft_ms": w["slo_ttft_ms"][m: m + 1]}
    if "events" in w:
        ev = w["events"]
        rows = np.flatnonzero(ev["req_model"] == m)
        keep = ev["model"] == m
        req = np.searchsorted(rows, ev["req"][keep]).astype(np.int32)
        one["events"] = {"model": np.zeros(int(keep.sum()), np.int32), "req": req,
                         "t_s": ev["t_s"][keep], "phase": ev["phase"][keep],
                         "req_model": np.zeros(len(rows), np.int32),
                         "req_t_arr_ms": ev["req_t_arr_ms"][rows],
                         "req_ttft_ms": ev["req_ttft_ms"][rows]}
    else:
        keep = w["requests"]["model"] == m
        one["requests"] = {k: (np.zeros(int(keep.sum()), np.int32) if k == "model" else v[keep])
                           for k, v in w["requests"].items()}
    return one


def _oracle_model_unit(args):
    one, dtype = args
    prof = tracegen.default_profile(1, one["window_ms"])
    return _oracle_models(one, np.dtype(dtype).type, prof)


def _noop(x):
    return x


def config_cpu(w, dtype, frac, pool):
    """The oracle's rate on a bounded sample of a workload (the first `frac` of
    its duration): single-threaded, and with its models as independent units
    over the worker pool (reduce, calibrate and score per model) followed by
    the walk."""
    import oracle
    sw = cut_workload(w, frac)
    n = len(sw["events"]["model"]) if "events" in sw else len(sw["requests"]["model"])
    npdt = np.float32 if dtype == "f32" else np.float64
    t0 = time.perf_counter()
    _oracle_path(sw, npdt)
    dt1 = time.perf_counter() - t0
    what = (f"first {sw['K'] * sw['window_ms'] / 1000:.0f} s of the trace ({n} "
            f"{'token events' if 'events' in sw else 'request records'}, {sw['K']} windows)")
    res = {"value": n / dt1, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": what,
           "seconds": dt1}
    if pool is not None:
        try:
            t0 = time.perf_counter()
            parts = pool.map_async(_oracle_model_unit,
                                   [(_model_slice(sw, m), np.dtype(npdt).name)
                                    for m in range(sw["M"])], chunksize=1).get(timeout=600)
            Z = np.stack([p[0][:, 0] for p in parts], 1)
            cls = np.stack([p[1][:, 0] for p in parts], 1)
            oracle.select_moves(Z, cls, 0.8, 1.2, sw["window_ms"], sw["budget"], sw["r0"],
                                sw["r_min"], sw["footprint"], sw["fast_ms"], sw["slow_ms"],
                                sw["pacing_cap"])
            dtp = time.perf_counter() - t0
            res["parallel"] = {"value": n / dtp, "unit": UNIT, "cores": pool._processes,
                               "kind": "oracle", "seconds": dtp,
                               "sample": what + f"; {sw['M']} per-model units over "
                                                f"{pool._processes} processes, then the walk"}
        except Exception as e:   # a baseline must not cost the bench line
            res["parallel"] = {"error": f"{type(e).__name__}: {e}"}
    return res


def measure_configs(tre, lib, Trace, hbm, peak_kind, with_cpu):
    """Device time of one pass of the whole path per workload and dtype, with
    L2 flushed (a buffer of twice its size written) before every step and the
    step alone between the CUDA events; phase times from the library's
    events; the oracle's rates beside it."""
    import multiprocessing as mp

    import torch
    pool = None
    if with_cpu:
        try:
            pool = mp.get_context("spawn").Pool(max(1, os.cpu_count() or 1))
            pool.map_async(_noop, range(pool._processes)).get(timeout=120)
        except Exception:
            pool = None
    l2 = torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size
    flush = torch.empty(2 * max(int(l2), 1 << 20), dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    out = {}
    try:
        for key, name, dtypes, steps, frac in CONFIGS:
            w = tracegen.workload(name, scale=1.0)
            dev = ({"events": {k: torch.as_tensor(v).cuda() for k, v in w["events"].items()}}
                   if "events" in w else
                   {"requests": {k: torch.as_tensor(v).cuda() for k, v in w["requests"].items()}})
            prof = tracegen.default_profile(w["M"], w["window_ms"])
            n_units = len(w["events"]["model"]) if "events" in w else len(w["requests"]["model"])
            tokens = int(w["requests"]["L_in"].astype(np.int64).sum() +
                         w["requests"]["L_out"].astype(np.int64).sum())
            entry = {"records_or_events": n_units,
                     "unit_kind": "token events" if "events" in w else "request records",
                     "model_windows": w["K"] * w["M"], "tokens": tokens, "dtypes": {}}
            for dt in dtypes:
                plan = tre.PipelinePlan(w["M"], w["window_ms"], w["K"], prof, w["slo_ttft_ms"],
                                        w["budget"], w["r0"], w["r_min"], w["footprint"],
                                        dtype=dt, fast_ms=w["fast_ms"], slow_ms=w["slow_ms"],
                                        pacing_cap=w["pacing_cap"], moves_cap=1 << 16, **dev)
                for _ in range(3):
                    plan.run(stream)
                torch.cuda.synchronize()
                lib.tre_trace_enable(1)
                evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(steps)]
                for a, b in evs:
                    flush.fill_(1)
                    a.record(stream)
                    plan.run(stream)
                    b.record(stream)
                torch.cuda.synchronize()
                tr = Trace()
                lib.tre_trace_collect(C.byref(tr))
                lib.tre_trace_enable(0)
                ms = sum(a.elapsed_time(b) for a, b in evs) / steps
                tsize = 4 if dt == "f32" else 8
                byts = config_bytes(w, tsize)
                ph = {tr.name[i].decode(): tr.ms[i] / steps * 1e3 for i in range(tr.n_phases)
                      if tr.calls[i]}
                launches = int(sum(tr.launches[i] for i in range(tr.n_phases))) // steps
                achieved = byts / (ms / 1e3) / 1e9
                e = {"us_per_step": ms * 1e3, "steps": steps,
                     "events_per_s": n_units / (ms / 1e3),
                     "model_windows_per_s": w["K"] * w["M"] / (ms / 1e3),
                     "tokens_per_s": tokens / (ms / 1e3), "n_moves": int(plan.n_moves.item()),
                     "algorithmic_bytes": byts,
                     "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm,
                                  "unit": "GB/s", "frac": achieved / hbm,
                                  "peak_kind": peak_kind},
                     "phases_us_per_step": ph, "launches_per_step": launches,
                     "l2": "flushed before every step (2x L2 written)"}
                if with_cpu:
                    e["cpu_baseline"] = config_cpu(w, dt, frac, pool)
                entry["dtypes"][dt] = e
                del plan
            out[key] = entry
            del dev, w
            torch.cuda.empty_cache()
    finally:
        if pool is not None:
            pool.terminate()
    return out


TRACE_PHASES = 11   # phases of tre_trace (the library header's count)


def occupancy_cpu(scale):
    """The oracle's time-averaged occupancy on one trace of the workload (1 core)."""
    import oracle
    sw = tracegen.sweep_workload(scale=scale, n_traces=1)
    req = sw["traces"][0]
    t0 = time.perf_counter()
    oracle.occupancy_mean_requests(req, sw["M"], 100, sw["duration_ms"] // 100)
    dt = time.perf_counter() - t0
    n = len(req["model"])
    return {"value": n / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"1 trace ({n} records) at the 100 ms grid; {dt:.2f} s"}


def occupancy_measure(lib, Trace, dev_traces, M, duration_ms, hbm, peak_kind, reps=5):
    """The time-averaged occupancy pass of tss_window_reduce (request-ms running
    and waiting per window) on each trace of the workload at the 100 ms grid,
    timed on the device by the library's phase events. The seven traces are
    taken in turn (196 MB of records in all, more than L2), so a trace's columns
    are not resident when it comes round again."""
    import torch

    import paper_2609_29160_gb300 as tre
    win = 100
    K = duration_ms // win
    out = {k: torch.empty((K, M), dtype=torch.int32, device="cuda") for k in "PDAW"}
    for k in ("A_ms", "W_ms"):
        out[k] = torch.empty((K, M), dtype=torch.int64, device="cuda")
    diag = tre.new_diag()
    for t in dev_traces:
        tre.tss_window_reduce(M, win, K, requests=t, out=out, diag=diag, mean_occupancy=True)
    torch.cuda.synchronize()
    lib.tre_trace_enable(1)
    for _ in range(reps):
        for t in dev_traces:
            tre.tss_window_reduce(M, win, K, requests=t, out=out, diag=diag, mean_occupancy=True)
    torch.cuda.synchronize()
    tr = Trace()
    lib.tre_trace_collect(C.byref(tr))
    lib.tre_trace_enable(0)
    ph = {tr.name[i].decode(): (tr.ms[i], tr.calls[i]) for i in range(tr.n_phases)}
    n_rec = sum(int(t["model"].numel()) for t in dev_traces) / len(dev_traces)
    occ_ms, occ_calls = ph["occupancy"]
    red_ms, red_calls = ph["reduce"]
    us = occ_ms / max(occ_calls, 1) * 1e3
    # algorithmic bytes: the records' columns read once, the two int64 outputs
    # written once
    byts = n_rec * 28 + K * M * 16
    achieved = byts / (us / 1e6) / 1e9
    return {"row": "time-averaged running/waiting occupancy (request-ms per window)",
            "window_ms": win, "records_per_call": int(n_rec), "model_windows_per_call": K * M,
            "us_per_call": us, "sampled_reduce_us_per_call": red_ms / max(red_calls, 1) * 1e3,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                         "frac": achieved / hbm, "peak_kind": peak_kind,
                         "bytes_per_call": byts, "traffic": None},
            "l2": "7 traces in turn, 196 MB of records"}


# ---------------------------------------------------------------------------
# Closed-loop replay of the sweep's traces (a widened row beside the sweep)
# ---------------------------------------------------------------------------
REPLAY_WAKE_MS, REPLAY_SLEEP_MS = 1310, 1870     # measured wake / sleep averages


def replay_measure(lib, Trace, sw, theta, scale, rank, passes=2):
    """tre_replay for every (trace, window length) of the sweep with all 64
    (rescue threshold, pacing cap) settings each -- 1792 closed-loop controller
    instances -- with the measured wake and sleep delays, a latency guard at
    twice each model's TTFT bound, and theta as the open-loop sweep calibrated
    it. Device time per pass over the 28 calls (the seven traces on seven
    streams side by side, CUDA events around the pass), and the TTFT
    attainment of the paper's rule (threshold 0.8, one transition per tick)
    and of the best and worst settings per window length."""
    import torch

    import paper_2609_29160_gb300 as tre
    M = sw["M"]
    dur = sw["duration_ms"]
    slo = np.asarray(sw["slo_ttft_ms"], np.int32)
    taus, caps = [float(t) for t in sw["tau_crit"]], [int(c) for c in sw["pacing_cap"]]
    plans, meta = [], []
    n_tr = len(sw["traces"])
    th = theta.cpu().numpy()
    for ti in range(n_tr):
        spec = tracegen.spec_mid(scale, sw["trace_seeds"][ti], dur / 1000.0)
        lat = tracegen.gen_latent(spec)
        dev = {k: torch.as_tensor(lat[k]).cuda() for k in tre.LATENT_KEYS}
        for wi, win in enumerate(sw["window_ms"]):
            win = int(win)
            prof = {"w_p": sw["w_p"], "w_q": sw["w_q"], "alpha": min(1.0, win / 5000.0),
                    "theta": th[ti * len(sw["window_ms"]) + wi], "tau_crit": 0.8,
                    "tau_surplus": sw["tau_surplus"]}
            plans.append(tre.ReplayPlan(dev, M, win, dur // win, prof, sw["budget"], lat["r0"],
                                        sw["r_min"], sw["footprint"], tau_list=taus,
                                        cap_list=caps, wake_ms=REPLAY_WAKE_MS,
                                        sleep_ms=REPLAY_SLEEP_MS, slo_ttft_ms=slo,
                                        guard_ttft_ms=2 * slo, dtype="f32", moves_cap=1024))
            meta.append((ti, win, len(lat["model"]), dur // win))
    # one stream per trace: a trace's four window lengths in turn, the traces
    # side by side
    main = torch.cuda.current_stream()
    streams = [torch.cuda.Stream() for _ in range(n_tr)]

    def one_pass():
        ev = torch.cuda.Event()
        ev.record(main)
        done = []
        for ti, st in enumerate(streams):
            st.wait_event(ev)
            for p, mt in zip(plans, meta):
                if mt[0] == ti:
                    p.run(st)
            d = torch.cuda.Event()
            d.record(st)
            done.append(d)
        for d in done:
            main.wait_event(d)

    one_pass()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(main)
    for _ in range(passes):
        one_pass()
    e1.record(main)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / passes
    n_inst = sum(p.n_inst for p in plans)
    inst_windows = sum(p.n_inst * k for p, (_, _, _, k) in zip(plans, meta))
    records = sum(n for (_, _, n, _) in meta)
    att = {}
    for win in sw["window_ms"]:
        win = int(win)
        met = np.zeros((len(taus) * len(caps),), np.float64)
        tot = 0
        for p, (ti, w, n, _) in zip(plans, meta):
            if w != win:
                continue
            met += p.out["slo_met"].cpu().numpy().sum(axis=1)
            tot += n
        a = met / max(tot, 1)
        rule = taus.index(0.8) * len(caps) + caps.index(1)
        best = int(np.argmax(a))
        att[str(win)] = {"paper_rule": float(a[rule]), "best": float(a[best]),
                         "best_setting": {"tau_crit": taus[best // len(caps)],
                                          "pacing_cap": caps[best % len(caps)]},
                         "worst": float(a.min())}
    return {"row": "closed-loop replay: 7 traces x 4 window lengths x 64 settings",
            "instances": n_inst, "ms_per_pass": ms, "calls_per_pass": len(plans),
            "instance_windows_per_s": inst_windows / (ms / 1e3),
            "records_per_s": records * len(taus) * len(caps) / (ms / 1e3),
            "wake_ms": REPLAY_WAKE_MS, "sleep_ms": REPLAY_SLEEP_MS,
            "guard": "2 x TTFT bound", "ttft_attainment": att,
            "bound": "latency (one warp per instance, serial over windows)"}


# DRAM traffic per call of a phase, from the committed ncu summary of its
# kernels; used only while the kernel source is the one the counters were
# taken on (the summary records its SHA-256)
TRAFFIC_SUMMARIES = {"reduce": ("profiles/k_reduce_requests_sweep_7x1M.md",
                                "paper_2609_29160_gb300/csrc/reduce.cu")}


def captured_traffic(phase):
    """DRAM bytes per call of a phase's kernel as one ncu capture measured them
    (not measured in this run): taken from the committed capture summary, and
    only while the kernel's source is the one the counters were taken on."""
    import hashlib
    import re
    if phase not in TRAFFIC_SUMMARIES:
        return None
    rel_summ, rel_src = TRAFFIC_SUMMARIES[phase]
    summ, src = os.path.join(ROOT, rel_summ), os.path.join(ROOT, rel_src)
    try:
        fields = {}
        for line in open(summ):
            hit = re.match(r"^[-*\s]*(dram_bytes_per_call|source_sha256):\s*`?([0-9a-f]+)`?", line)
            if hit:
                fields[hit.group(1)] = hit.group(2)
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
        if fields.get("source_sha256") != digest:
            return None
        return {"dram_bytes_per_call": float(fields["dram_bytes_per_call"]), "summary": rel_summ}
    except (OSError, KeyError, ValueError):
        return None


def phase_bytes(sw, n_records_per_trace, M):
    """Algorithmic bytes of one call of each phase over the whole sweep: what the
    method must read and write once, per record and per (window, model)."""
    nt = len(sw["traces"])
    K = [sw["duration_ms"] // int(w) for w in sw["window_ms"]]
    Kb = sw["duration_ms"] // int(min(sw["window_ms"]))
    mw = sum(K) * nt * M                      # model-windows over all series
    base = Kb * M * nt                        # base-grid cells over all traces
    return {
        # 7 int32 columns per record in; P, D, A/W diffs (4 B each) and the
        # packed SLO counts (8 B) per base cell out
        "reduce": float(np.sum(n_records_per_trace)) * 28 + base * 24,
        # gauge diffs in (block sums and their prefixes)
        "gauge_scan": base * 8,
        # diffs, base counts and SLO in; base gauges and every coarser
        # series' counts, gauges and SLO out
        "aggregate": base * (8 + 16) + base * 8 + (mw - base) * 24,
        # counts in, S and the idle flag out
        "score": mw * (16 + 4 + 1),
        # S, idle flag and SLO counts in
        "calibrate": mw * (4 + 1 + 8),
        # S and idle flag in, Z and region out
        "normalize": mw * (4 + 1 + 4 + 1),
    }


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    import torch
    import torch.distributed as dist

    import paper_2609_29160_gb300 as tre

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")
    lib = tre.load()
    lib.tre_trace_enable.argtypes = [C.c_int]

    NP = TRACE_PHASES

    class Trace(C.Structure):
        _fields_ = [("n_phases", C.c_int32), ("name", C.c_char_p * NP), ("ms", C.c_double * NP),
                    ("calls", C.c_int64 * NP), ("launches", C.c_int64 * NP)]
    lib.tre_trace_collect.argtypes = [C.POINTER(Trace)]

    # the seven traces are independent problems: rank r sweeps traces
    # t % world == r, so N ranks share one job (strong scaling); a rank
    # without a trace only takes part in the collectives
    from paper_2609_29160_gb300 import partition
    sw = tracegen.sweep_workload(scale=args.scale, seed0=SWEEP_SEED0)
    mine = partition.sweep_traces(len(sw["traces"]), rank, world)
    sw["trace_seeds"] = [SWEEP_SEED0 + t for t in mine]
    sw["traces"] = [sw["traces"][t] for t in mine]
    if not mine:
        return idle_rank(dist, world)
    M = sw["M"]
    win = sw["window_ms"]
    al = alphas(win)
    n_rec = [len(t["model"]) for t in sw["traces"]]
    total_rec = int(sum(n_rec))
    K = [sw["duration_ms"] // int(w) for w in win]
    model_windows = sum(K) * len(sw["traces"]) * M
    n_inst = len(sw["traces"]) * len(win) * len(sw["tau_crit"]) * len(sw["pacing_cap"])
    # prompt + output tokens of the step's records, and windows walked by all
    # controller instances
    tokens = int(sum(int(t["L_in"].astype(np.int64).sum() + t["L_out"].astype(np.int64).sum())
                     for t in sw["traces"]))
    inst_windows = len(sw["traces"]) * len(sw["tau_crit"]) * len(sw["pacing_cap"]) * sum(K)
    moves_cap = 512
    dev_traces = [{k: torch.as_tensor(v).cuda() for k, v in t.items()} for t in sw["traces"]]
    torch.cuda.synchronize()
    # a stream of its own: a CUDA graph cannot be captured on the default stream
    stream = torch.cuda.Stream()

    # the call is marshalled once; each step is one tre_sweep call on the stream
    plan = tre.SweepPlan(dev_traces, M, sw["duration_ms"], win, al, sw["tau_crit"],
                         sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                         sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"], sw["footprint"],
                         dtype="f32", moves_cap=moves_cap)

    def step():
        return plan.run(stream)

    for _ in range(args.warmup):
        out = step()
    torch.cuda.synchronize()

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    l2 = torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size
    # Inputs larger than L2 (the whole sweep on one GPU: 196 MB) need no flush;
    # the timed steps are then one CUDA graph of the K calls, replayed once.
    # A rank holding less than that (several GPUs split the traces) flushes L2
    # before every step (twice its size written), outside the step's events.
    in_bytes = int(sum(v.numel() * v.element_size() for t in dev_traces for v in t.values()))
    use_graph = in_bytes >= int(1.25 * l2) and not args.no_graph
    graph = traced = None

    def capture(trace_on):
        lib.tre_trace_enable(1 if trace_on else 0)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream, capture_error_mode="relaxed"):
            for _ in range(args.steps):
                step()
        with torch.cuda.stream(stream):
            g.replay()                   # warm-up replay
        torch.cuda.synchronize()
        return g

    if use_graph:
        try:
            # the timed graph carries no phase events; a second graph of the
            # same calls with the library's phase events is replayed after it
            graph = capture(False)
            traced = capture(True)       # tracing stays on: its events are the phases'
        except Exception as e:           # capture refused: time the calls one by one
            graph = traced = None
            graph_error = f"{type(e).__name__}: {e}"
            lib.tre_trace_enable(0)
    if graph is None:
        lib.tre_trace_enable(1)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    c0 = clocks.now()
    if graph is not None:
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        with torch.cuda.stream(stream):
            graph.replay()
        ev1.record(stream)
        torch.cuda.synchronize()
        ms = ev0.elapsed_time(ev1)
    else:
        flush = torch.empty(2 * max(int(l2), 1 << 20), dtype=torch.uint8, device="cuda")
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(args.steps)]
        for a, b in evs:
            with torch.cuda.stream(stream):
                flush.fill_(1)
            a.record(stream)
            out = step()
            b.record(stream)
        torch.cuda.synchronize()
        ms = sum(a.elapsed_time(b) for a, b in evs)
    c1 = clocks.now()
    if world > 1:
        dist.barrier()
    if traced is not None:
        with torch.cuda.stream(stream):
            traced.replay()              # the phases of the same K calls
        torch.cuda.synchronize()
    tr = Trace()
    lib.tre_trace_collect(C.byref(tr))
    lib.tre_trace_enable(0)
    timing = {"launch": "one CUDA graph of the timed calls (phase times from a replay of a "
                        "second graph of the same calls with the library's phase events)"
              if graph is not None else "calls one by one, L2 flushed before each",
              "input_bytes": in_bytes, "l2_bytes": int(l2)}
    if use_graph and graph is None:
        timing["graph_error"] = graph_error
    # the same step, back to back for at least 1.5 s right after the timed
    # region: long enough for the 100 ms clock samples to see the kernels
    n_sus = max(1, int(1500.0 / max(ms / args.steps, 1e-3)) + 1)
    es0, es1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0 = clocks.now()
    es0.record(stream)
    if graph is not None:
        reps = max(1, n_sus // args.steps)
        with torch.cuda.stream(stream):
            for _ in range(reps):
                graph.replay()
        n_sus = reps * args.steps
    else:
        for _ in range(n_sus):
            step()
    es1.record(stream)
    torch.cuda.synchronize()
    s1 = clocks.now()
    time.sleep(0.2)
    clocks.stop()
    clk = clocks.window(c0, s1, "timed region and the sustained loop of the same step after it")
    clk["timed_region_samples"] = clocks.window(c0, c1, "")["samples"]
    sustained = {"steps": n_sus, "ms_per_step": es0.elapsed_time(es1) / n_sus,
                 "clocks": clocks.window(s0, s1, "sustained loop only")}
    job_rec, job_mw, job_inst, job_tok, job_iw = (total_rec, model_windows, n_inst, tokens,
                                                  inst_windows)
    if world > 1:
        ms, (job_rec, job_mw, job_inst, job_tok, job_iw) = over_ranks(
            dist, "cuda", ms, [total_rec, model_windows, n_inst, tokens, inst_windows])
    ms_step = ms / args.steps
    value = job_rec * args.steps / (ms / 1e3)
    mw_s = job_mw * args.steps / (ms / 1e3)
    tok_s = job_tok * args.steps / (ms / 1e3)
    iw_s = job_iw * args.steps / (ms / 1e3)
    phases = {tr.name[i].decode(): {"ms": tr.ms[i], "calls": tr.calls[i],
                                    "launches": tr.launches[i]} for i in range(tr.n_phases)}
    launches = int(sum(p["launches"] for p in phases.values()))

    # dominant kernel phase and its roofline
    hbm, peak_kind = peaks()
    pb = phase_bytes(sw, n_rec, M)
    dom = max(phases, key=lambda k: phases[k]["ms"])
    share = phases[dom]["ms"] / max(ms, 1e-9)
    def roof_of(name):
        per_call_ms = phases[name]["ms"] / max(phases[name]["calls"], 1)
        achieved = pb[name] / (per_call_ms / 1e3) / 1e9
        cap = captured_traffic(name)
        # traffic: DRAM bytes per call from the one ncu capture of this kernel
        # source (null once the source has changed since the capture)
        return {"bound": "hbm", "kernel": name, "achieved": achieved, "peak": hbm,
                "unit": "GB/s", "frac": achieved / hbm,
                "traffic": cap["dram_bytes_per_call"] if cap else None,
                "ncu_capture": cap,
                "share_of_step": phases[name]["ms"] / max(ms, 1e-9), "peak_kind": peak_kind,
                "bytes_per_call": pb[name], "us_per_call": per_call_ms * 1e3}
    if dom in pb and phases[dom]["calls"]:
        roof = roof_of(dom)
    else:
        # the controller walk is serial over control ticks: no bandwidth roofline
        # applies; report the largest bandwidth-bound phase beside it
        hb = max((k for k in pb if phases.get(k, {}).get("calls")), key=lambda k: phases[k]["ms"])
        roof = roof_of(hb)
        roof["dominant_phase"] = {"name": dom, "share_of_step": share,
                                  "bound": "latency (serial over control ticks)"}
    # whole-step view against HBM: algorithmic bytes of the full sweep per step
    step_bytes = total_rec * 28 + model_windows * (16 + 4 + 4 + 1)
    whole = {"algorithmic_bytes": step_bytes, "achieved_gbs": step_bytes / (ms_step / 1e3) / 1e9,
             "frac": step_bytes / (ms_step / 1e3) / 1e9 / hbm}

    # End to end: every step takes its records from pinned host memory and
    # reads its results back. Where the GPU addresses pinned host memory
    # directly (unified addressing maps cudaHostAlloc'd memory at the same
    # address), the sweep reads the records from host memory itself; otherwise
    # the records are copied in as one block per step over four streams, the
    # next step's copy overlapping this step's sweep (two device buffers).
    keys = list(dev_traces[0].keys())
    host = [{k: v.cpu().pin_memory() for k, v in t.items()} for t in dev_traces]
    h2d = sum(v.numel() * v.element_size() for t in host for v in t.values())
    res_keys = ("n_moves", "r_final", "theta")
    n_e2e = max(args.e2e_steps, 2)
    if host_mapped(host[0][keys[0]].data_ptr()):
        # two marshalled calls on two streams: step i+1's reduction (bound by
        # reading the host records) overlaps step i's later phases
        mode = ("sweep reads the records from pinned host memory; consecutive steps on two "
                "streams")
        plans_h = [tre.SweepPlan(host, M, sw["duration_ms"], win, al, sw["tau_crit"],
                                 sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                                 sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"],
                                 sw["footprint"], dtype="f32", moves_cap=moves_cap)
                   for _ in range(2)]
        res_host = [{k: torch.empty_like(plans_h[0].out[k], device="cpu").pin_memory()
                     for k in res_keys} for _ in range(2)]
        d2h = sum(v.numel() * v.element_size() for v in res_host[0].values())
        strs = [stream, torch.cuda.Stream()]
        for j in range(2):
            plans_h[j].run(strs[j])
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        fin = torch.cuda.Event()
        e0.record(stream)
        strs[1].wait_event(e0)
        for i in range(n_e2e):
            j = i % 2
            plans_h[j].run(strs[j])
            with torch.cuda.stream(strs[j]):
                for k in res_keys:
                    res_host[j][k].copy_(plans_h[j].out[k], non_blocking=True)
        fin.record(strs[1])
        stream.wait_event(fin)
        e1.record(stream)
    else:
        mode = "records copied in per step (4 streams, overlapping the previous sweep)"
        offs, o = [], 0
        for t in dev_traces:
            offs.append({})
            for k in keys:
                offs[-1][k] = o
                o += (t[k].numel() * 4 + 15) // 16 * 16
        block = o
        host_blk = torch.empty(block, dtype=torch.uint8).pin_memory()
        for t, of in zip(host, offs):
            for k in keys:
                n = t[k].numel()
                host_blk[of[k]:of[k] + 4 * n].view(torch.int32).copy_(t[k])
        dev_blk = [torch.empty(block, dtype=torch.uint8, device="cuda") for _ in range(2)]
        views = [[{k: blk[of[k]:of[k] + 4 * t[k].numel()].view(torch.int32) for k in keys}
                  for t, of in zip(dev_traces, offs)] for blk in dev_blk]
        plans = [tre.SweepPlan(v, M, sw["duration_ms"], win, al, sw["tau_crit"],
                               sw["pacing_cap"], sw["w_p"], sw["w_q"], sw["tau_surplus"],
                               sw["slo_ttft_ms"], sw["budget"], sw["r0"], sw["r_min"],
                               sw["footprint"], dtype="f32", moves_cap=moves_cap) for v in views]
        h2d = block
        res_host2 = [{k: torch.empty_like(plans[0].out[k], device="cpu").pin_memory()
                      for k in res_keys} for _ in range(2)]
        d2h = sum(v.numel() * v.element_size() for v in res_host2[0].values())
        kParts = 4
        part = (block + kParts - 1) // kParts
        cuts = [(q * part, min(block, (q + 1) * part)) for q in range(kParts)]
        copy = torch.cuda.Stream()
        lanes = [torch.cuda.Stream() for _ in range(kParts)]
        lane_done = [torch.cuda.Event() for _ in range(kParts)]
        done = [torch.cuda.Event() for _ in range(n_e2e)]      # sweep i finished
        freed = [torch.cuda.Event() for _ in range(n_e2e)]     # buffer of step i free
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(copy)
        for i in range(n_e2e):
            j = i % 2
            with torch.cuda.stream(copy):
                if i >= 2:
                    copy.wait_event(done[i - 2])
                freed[i].record(copy)
            for (c0, c1), ln, ev in zip(cuts, lanes, lane_done):
                ln.wait_event(freed[i])
                with torch.cuda.stream(ln):
                    dev_blk[j][c0:c1].copy_(host_blk[c0:c1], non_blocking=True)
                    ev.record(ln)
            for ev in lane_done:
                stream.wait_event(ev)
            plans[j].run(stream)
            done[i].record(stream)
            with torch.cuda.stream(copy):
                copy.wait_event(done[i])
                for k in res_keys:
                    res_host2[j][k].copy_(plans[j].out[k], non_blocking=True)
        e1.record(copy)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1) / n_e2e
    if world > 1:
        e2e_ms, _ = over_ranks(dist, "cuda", e2e_ms, [])
    e2e = {"value": job_rec / (e2e_ms / 1e3), "unit": UNIT,
           "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
           "ms_per_step": e2e_ms, "steps": n_e2e, "mode": mode}

    # a widened step measured beside the sweep (not part of the timed step)
    next_rows = {"occupancy_mean": occupancy_measure(lib, Trace, dev_traces, M,
                                                     sw["duration_ms"], hbm, peak_kind)}
    if not args.no_replay:
        next_rows["closed_loop_replay"] = replay_measure(lib, Trace, sw, out["theta"],
                                                         args.scale, rank)

    configs = None
    if rank == 0 and not args.no_configs:
        configs = measure_configs(tre, lib, Trace, hbm, peak_kind,
                                  with_cpu=world == 1 and not args.no_cpu_baseline)

    base = base_par = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        base = cpu_baseline(args.scale)
        base["host"] = host_cpu()
        next_rows["occupancy_mean"]["cpu_baseline"] = occupancy_cpu(args.scale)
        base_par = cpu_baseline_parallel(args.scale, SWEEP_SEED0)
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "strong", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic",
            "config": {"workload": WORKLOAD, "records_per_step": int(job_rec),
                       "model_windows_per_step": int(job_mw),
                       "controller_instances": int(job_inst), "scale": args.scale,
                       "l2": "inputs larger than L2 (7 x 28 B x ~1M records = 196 MB) on one "
                             "GPU; a rank with less flushes L2 before every step (2x L2 "
                             "written, outside the timed events)",
                       "parallelism": f"the sweep's 7 traces split over {world} GPU(s) "
                                      "(trace t on rank t % N)"},
            "model_windows_per_s": mw_s, "tokens_per_s": tok_s,
            "instance_windows_per_s": iw_s,
            "roofline": roof, "step_roofline": whole, "phases_ms_per_step": {
                k: p["ms"] / args.steps for k, p in phases.items() if p["calls"]},
            "phases_roofline": {k: round(roof_of(k)["frac"], 4) for k in pb
                                if phases.get(k, {}).get("calls")},
            "gpu_launches": launches, "clocks": clk, "sustained": sustained, "timing": timing,
            "e2e": e2e,
            "cpu_baseline": base,
            "cpu_baseline_parallel": base_par,
            "next_rows": next_rows, "configs": configs,
        }
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
