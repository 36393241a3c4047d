"""GB300 Token Service Share / TRE library: thin Python binding of libtre.so.

Functions here carry the names of the C ABI in include/tre.h and only marshal
arguments: torch CUDA tensors become device pointers, the current torch stream
becomes the launch stream, and workspaces are allocated with torch. Every step
of the computation runs in the library's CUDA kernels; there is no fallback, and
loading fails loudly when the compiled library is missing.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from . import _build

CRIT, NOM, SURP, IDLE = 0, 1, 2, 3
RESCUE, REBALANCE = 1, 2
F32, F64 = 0, 1
STATUS = {0: "ok", 1: "invalid argument", 2: "workspace too small", 3: "CUDA error",
          4: "move list overflow", 5: "device wait timed out"}


class TreError(RuntimeError):
    def __init__(self, fn, code):
        super().__init__(f"{fn}: {STATUS.get(code, code)} ({code})")
        self.code = code


class Grid(C.Structure):
    _fields_ = [("n_models", C.c_int32), ("window_ms", C.c_int32), ("n_windows", C.c_int32)]


class Requests(C.Structure):
    _fields_ = [("n", C.c_int64)] + [(k, C.c_void_p) for k in (
        "model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")]


class Events(C.Structure):
    _fields_ = [("n", C.c_int64), ("model", C.c_void_p), ("req", C.c_void_p),
                ("t_s", C.c_void_p), ("phase", C.c_void_p), ("n_req", C.c_int64),
                ("req_model", C.c_void_p), ("req_t_arr_ms", C.c_void_p),
                ("req_ttft_ms", C.c_void_p)]


class Counts(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("P", "D", "A", "W", "A_ms", "W_ms")]


class Profile(C.Structure):
    _fields_ = [("dtype", C.c_int)] + [(k, C.c_void_p) for k in (
        "w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")]


class Ctrl(C.Structure):
    _fields_ = [("budget", C.c_int64), ("r_min", C.c_void_p), ("footprint", C.c_void_p),
                ("fast_ms", C.c_int32), ("slow_ms", C.c_int32), ("pacing_cap", C.c_int32)]


class Diag(C.Structure):
    _fields_ = [("dropped_range", C.c_uint64), ("dropped_model", C.c_uint64),
                ("dropped_order", C.c_uint64), ("degenerate_calib", C.c_uint64),
                ("ema_resolved", C.c_uint64), ("err", C.c_int32), ("reserved", C.c_int32)]


class SweepSpec(C.Structure):
    _fields_ = [("n_models", C.c_int32), ("duration_ms", C.c_int32), ("n_traces", C.c_int32),
                ("traces", C.POINTER(Requests)), ("n_win", C.c_int32),
                ("window_ms", C.POINTER(C.c_int32)), ("alpha", C.POINTER(C.c_double)),
                ("n_tau", C.c_int32), ("tau_crit", C.POINTER(C.c_double)), ("n_cap", C.c_int32),
                ("pacing_cap", C.POINTER(C.c_int32)), ("dtype", C.c_int),
                ("w_p", C.c_void_p), ("w_q", C.c_void_p), ("tau_surplus", C.c_void_p),
                ("slo_ttft_ms", C.c_void_p), ("ok_frac", C.c_double),
                ("reliability", C.c_double), ("ctrl", Ctrl), ("r0", C.c_void_p)]


class SweepOut(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("P", "D", "A", "W", "S", "Z", "cls", "theta", "moves")] + [
        ("moves_cap", C.c_int64), ("n_moves", C.c_void_p), ("r_final", C.c_void_p)]


class Latent(C.Structure):
    _fields_ = [("n", C.c_int64)] + [(k, C.c_void_p) for k in (
        "model", "t_arr_ms", "d_first_ms", "d_total_ms", "L_in", "L_out")]


class ReplaySpec(C.Structure):
    _fields_ = [("n_tau", C.c_int32), ("tau_crit", C.POINTER(C.c_double)), ("n_cap", C.c_int32),
                ("pacing_cap", C.POINTER(C.c_int32)), ("wake_ms", C.c_int32),
                ("sleep_ms", C.c_int32), ("guard_ttft_ms", C.c_void_p)]


class ReplayOut(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("t_start_ms", "t_first_ms", "t_end_ms", "Z", "cls",
                                          "moves")] + [
        ("moves_cap", C.c_int64), ("n_moves", C.c_void_p), ("r_final", C.c_void_p),
        ("slo_met", C.c_void_p), ("served", C.c_void_p)]


MOVE_DTYPE = np.dtype([("window", np.int32), ("recv", np.int16), ("donor", np.int16),
                       ("kind", np.uint8), ("seq", np.uint8), ("reserved", np.uint16)])
DIAG_BYTES = C.sizeof(Diag)

_lib = None
EXPORTS = ("tss_window_reduce", "tss_score", "tss_calibrate", "tre_select_moves", "tre_sweep",
           "tre_status_str")


def library_path():
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libtre.so (building it in-tree first if asked). Raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if build_if_missing:
        path = _build.build()
    if not os.path.exists(path):
        raise RuntimeError(f"libtre.so not built ({path}); run __graft_entry__.build()")
    lib = C.CDLL(path)
    P = C.c_void_p
    lib.tss_window_reduce.argtypes = [C.POINTER(Grid), C.POINTER(Requests), C.POINTER(Events),
                                      Counts, P, C.POINTER(C.c_size_t), P, P]
    lib.tss_score.argtypes = [C.POINTER(Grid), C.POINTER(Counts), C.POINTER(Profile), P, P, P, P,
                              P, P, P, C.POINTER(C.c_size_t), P, P]
    lib.tss_calibrate.argtypes = [C.POINTER(Grid), C.POINTER(Requests), C.POINTER(Events),
                                  C.POINTER(Counts), C.POINTER(Profile), P, C.c_double,
                                  C.c_double, P, P, P, P, C.POINTER(C.c_size_t), P, P]
    lib.tss_normalize.argtypes = [C.POINTER(Grid), C.POINTER(Profile), P, P, P, P, P, P]
    lib.tre_select_moves.argtypes = [C.POINTER(Grid), P, P, C.POINTER(Profile), C.POINTER(Ctrl),
                                     P, P, C.c_int64, P, P, C.POINTER(C.c_size_t), P, P]
    lib.tre_sweep.argtypes = [C.POINTER(SweepSpec), C.POINTER(SweepOut), P,
                              C.POINTER(C.c_size_t), P, P]
    lib.tss_rank.argtypes = [C.POINTER(Grid), C.c_int, P, P, P, P, P]
    lib.tss_class_models.argtypes = [C.c_int64, P, P, C.c_int32, C.c_int32, P, P]
    lib.tss_class_models.restype = C.c_int
    lib.tss_stage_gauges.argtypes = [C.POINTER(Grid), C.POINTER(Requests), P, P, P,
                                     C.POINTER(C.c_size_t), P, P]
    lib.tss_stage_calibrate.argtypes = [C.POINTER(Grid), C.POINTER(Requests), C.POINTER(Counts),
                                        P, P, C.POINTER(Profile), P, P, C.c_double, C.c_double,
                                        P, P, P, C.POINTER(C.c_size_t), P, P]
    lib.tss_stage_score.argtypes = [C.POINTER(Grid), C.POINTER(Counts), P, P, C.POINTER(Profile),
                                    P, P, P, P, P, P, P, P, P, C.POINTER(C.c_size_t), P, P]
    for f in ("tss_window_reduce", "tss_score", "tss_calibrate", "tre_select_moves", "tre_sweep",
              "tss_rank", "tss_stage_gauges", "tss_stage_calibrate", "tss_stage_score",
              "tss_normalize"):
        getattr(lib, f).restype = C.c_int
    lib.tre_replay.argtypes = [C.POINTER(Grid), C.POINTER(Latent), C.POINTER(Profile),
                               C.POINTER(Ctrl), P, C.POINTER(ReplaySpec), P,
                               C.POINTER(ReplayOut), P, C.POINTER(C.c_size_t), P, P]
    lib.tre_replay.restype = C.c_int
    lib.tre_status_str.argtypes = [C.c_int]
    lib.tre_status_str.restype = C.c_char_p
    _lib = lib
    return lib


# ---------------------------------------------------------------------------
# torch plumbing
# ---------------------------------------------------------------------------
def _torch():
    import torch
    return torch


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _stream(stream):
    torch = _torch()
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def _check(fn, code):
    if code != 0:
        raise TreError(fn, code)


def _dt(dtype):
    torch = _torch()
    if dtype in (torch.float32, np.float32, "f32", F32):
        return F32, torch.float32
    if dtype in (torch.float64, np.float64, "f64", F64):
        return F64, torch.float64
    raise ValueError(dtype)


def new_diag(device="cuda"):
    """Zeroed device-resident tre_diag."""
    torch = _torch()
    return torch.zeros(DIAG_BYTES, dtype=torch.uint8, device=device)


def read_diag(diag):
    raw = diag.cpu().numpy().tobytes()
    d = Diag.from_buffer_copy(raw)
    return {k: getattr(d, k) for k, _ in Diag._fields_ if k != "reserved"}


def _workspace(fn, call):
    """Query the workspace size (ws=NULL), allocate it with torch, then call."""
    torch = _torch()
    size = C.c_size_t(0)
    _check(fn, call(None, C.byref(size)))
    ws = torch.empty(max(int(size.value), 256), dtype=torch.uint8, device="cuda")
    _check(fn, call(_ptr(ws), C.byref(size)))
    return ws


def _need(t, dtype, n=None, what="array"):
    """Checks a tensor argument before its pointer is handed to the library:
    element type, contiguity and (when given) element count."""
    torch = _torch()
    want = getattr(torch, dtype)
    if t.dtype != want:
        raise ValueError(f"{what}: expected {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{what}: must be contiguous")
    if n is not None and int(t.numel()) != n:
        raise ValueError(f"{what}: expected {n} elements, got {int(t.numel())}")


def requests_struct(req):
    """tre_requests from a dict of int32 tensors, CUDA or pinned host (keeps no
    reference)."""
    keys = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")
    n = int(req["model"].numel())
    for k in keys:
        _need(req[k], "int32", n, k)
    return Requests(n, *[req[k].data_ptr() if n else None for k in keys])


def events_struct(ev):
    n, nr = int(ev["model"].numel()), int(ev["req_model"].numel())
    for k, dt, cnt in (("model", "int32", n), ("req", "int32", n), ("t_s", "float32", n),
                       ("phase", "uint8", n), ("req_model", "int32", nr),
                       ("req_t_arr_ms", "int32", nr), ("req_ttft_ms", "int32", nr)):
        _need(ev[k], dt, cnt, k)
    return Events(n, ev["model"].data_ptr() if n else None, ev["req"].data_ptr() if n else None,
                  ev["t_s"].data_ptr() if n else None, ev["phase"].data_ptr() if n else None, nr,
                  ev["req_model"].data_ptr() if nr else None,
                  ev["req_t_arr_ms"].data_ptr() if nr else None,
                  ev["req_ttft_ms"].data_ptr() if nr else None)


def _counts(c):
    n = int(c["P"].numel())
    for k in ("P", "D", "A", "W"):
        _need(c[k], "int32", n, k)
    for k in ("A_ms", "W_ms"):
        if c.get(k) is not None:
            _need(c[k], "int64", n, k)
    occ = [c[k].data_ptr() if c.get(k) is not None else None for k in ("A_ms", "W_ms")]
    return Counts(*[c[k].data_ptr() for k in ("P", "D", "A", "W")], *occ)


def _profile(prof, M, tdt, code):
    torch = _torch()
    out = {}
    for k in ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus"):
        v = prof.get(k)
        if v is None:
            out[k] = None
            continue
        t = v if torch.is_tensor(v) else torch.as_tensor(np.broadcast_to(np.asarray(v), (M,)).copy())
        out[k] = t.to(device="cuda", dtype=tdt).contiguous()
    st = Profile(code, *[out[k].data_ptr() if out[k] is not None else None
                         for k in ("w_p", "w_q", "alpha", "theta", "tau_crit", "tau_surplus")])
    return st, out


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------
def tss_window_reduce(M, window_ms, K, requests=None, events=None, diag=None, stream=None,
                      out=None, mean_occupancy=False):
    """Per-window P, D, A, W ([K][M] int32 CUDA tensors) from request records or
    token events (dicts of CUDA tensors). With mean_occupancy also A_ms, W_ms:
    int64 request-milliseconds running / waiting per window; a dict holding
    them makes tss_score use the window means."""
    torch = _torch()
    lib = load()
    g = Grid(M, window_ms, K)
    if out is None:
        out = {k: torch.empty((K, M), dtype=torch.int32, device="cuda") for k in "PDAW"}
        if mean_occupancy:
            for k in ("A_ms", "W_ms"):
                out[k] = torch.empty((K, M), dtype=torch.int64, device="cuda")
    diag = new_diag() if diag is None else diag
    rq = requests_struct(requests) if requests is not None else None
    ev = events_struct(events) if events is not None else None
    cs = _counts(out)
    s = _stream(stream)
    _workspace("tss_window_reduce", lambda ws, n: lib.tss_window_reduce(
        C.byref(g), C.byref(rq) if rq else None, C.byref(ev) if ev else None, cs, ws, n,
        _ptr(diag), s))
    return out


def tss_score(counts, profile, window_ms, dtype="f32", carry=None, recv=True, diag=None,
              stream=None):
    """Eq. 1 -> EMA -> Eq. 2 -> regions. Returns dict S, Z, cls (and recv)."""
    torch = _torch()
    lib = load()
    K, M = counts["P"].shape
    code, tdt = _dt(dtype)
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    S = torch.empty((K, M), dtype=tdt, device="cuda")
    Z = torch.empty((K, M), dtype=tdt, device="cuda")
    cls = torch.empty((K, M), dtype=torch.uint8, device="cuda")
    rv = torch.empty(K, dtype=torch.int32, device="cuda") if recv else None
    diag = new_diag() if diag is None else diag
    cs = _counts(counts)
    s = _stream(stream)
    _workspace("tss_score", lambda ws, n: lib.tss_score(
        C.byref(g), C.byref(cs), C.byref(pst), _ptr(carry["S"]) if carry else None,
        _ptr(carry["init"]) if carry else None, _ptr(S), _ptr(Z), _ptr(cls), _ptr(rv), ws, n,
        _ptr(diag), s))
    return {"S": S, "Z": Z, "cls": cls, "recv": rv}


def tss_class_models(model, cls, n_models, n_classes, out=None, stream=None):
    """Per-(model, SLO class) ids (model * n_classes + class, -1 when out of
    range) as an int32 CUDA tensor, to pass as the records' model column with
    n_models * n_classes models."""
    torch = _torch()
    lib = load()
    n = int(model.numel())
    _need(model, "int32", None, "model")
    _need(cls, "int32", n, "cls")
    if out is None:
        out = torch.empty(n, dtype=torch.int32, device=model.device)
    _need(out, "int32", n, "out")
    _check("tss_class_models", lib.tss_class_models(C.c_int64(n), _ptr(model), _ptr(cls),
                                                    n_models, n_classes, _ptr(out),
                                                    _stream(stream)))
    return out


RANK_DONORS = 8


def tss_rank(Z, cls, window_ms=1000, recv=True, donors=True, stream=None):
    """Per window the Eq. 3 receiver and its first RANK_DONORS donors in release
    order (Sec. IV-B). Z, cls: CUDA tensors [K, M]. Returns dict recv [K] int32
    and donors [K, RANK_DONORS] int32 (-1 in unused slots)."""
    torch = _torch()
    lib = load()
    K, M = Z.shape
    code, _ = _dt(Z.dtype)
    g = Grid(M, window_ms, K)
    rv = torch.empty(K, dtype=torch.int32, device=Z.device) if recv else None
    dn = torch.empty((K, RANK_DONORS), dtype=torch.int32, device=Z.device) if donors else None
    Zc, cc = Z.contiguous(), cls.contiguous()
    _need(cc, "uint8", K * M, "cls")
    _check("tss_rank", lib.tss_rank(C.byref(g), code, _ptr(Zc), _ptr(cc), _ptr(rv), _ptr(dn),
                                    _stream(stream)))
    return {"recv": rv, "donors": dn}


def tss_stage_gauges(M, window_ms, K, requests, diag=None, stream=None):
    """Running requests split at the first token, read at each window's last
    millisecond: (A_prefill, A_decode) int32 [K][M] CUDA tensors."""
    torch = _torch()
    lib = load()
    g = Grid(M, window_ms, K)
    A_p = torch.empty((K, M), dtype=torch.int32, device="cuda")
    A_d = torch.empty((K, M), dtype=torch.int32, device="cuda")
    diag = new_diag() if diag is None else diag
    rq = requests_struct(requests)
    s = _stream(stream)
    _workspace("tss_stage_gauges", lambda ws, n: lib.tss_stage_gauges(
        C.byref(g), C.byref(rq), _ptr(A_p), _ptr(A_d), ws, n, _ptr(diag), s))
    return A_p, A_d


def tss_stage_calibrate(counts, A_prefill, A_decode, profile, window_ms, slo_ttft_ms,
                        slo_tpot_ms, requests, dtype="f32", ok_frac=0.95, reliability=0.95,
                        diag=None, stream=None):
    """theta of the prefill signal (against TTFT) and of the decode signal
    (against TPOT): two CUDA tensors of dtype [M]."""
    torch = _torch()
    lib = load()
    K, M = counts["P"].shape
    code, tdt = _dt(dtype)
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    i32 = lambda a: (a if torch.is_tensor(a) else torch.as_tensor(np.asarray(a, np.int32))).to(
        device="cuda", dtype=torch.int32).contiguous()
    ttft, tpot = i32(slo_ttft_ms), i32(slo_tpot_ms)
    for t, what in ((A_prefill, "A_prefill"), (A_decode, "A_decode")):
        _need(t, "int32", K * M, what)
    th_p = torch.empty(M, dtype=tdt, device="cuda")
    th_d = torch.empty(M, dtype=tdt, device="cuda")
    diag = new_diag() if diag is None else diag
    rq = requests_struct(requests)
    cs = _counts(counts)
    s = _stream(stream)
    _workspace("tss_stage_calibrate", lambda ws, n: lib.tss_stage_calibrate(
        C.byref(g), C.byref(rq), C.byref(cs), _ptr(A_prefill), _ptr(A_decode), C.byref(pst),
        _ptr(ttft), _ptr(tpot), C.c_double(ok_frac), C.c_double(reliability), _ptr(th_p),
        _ptr(th_d), ws, n, _ptr(diag), s))
    return th_p, th_d


def tss_stage_score(counts, A_prefill, A_decode, profile, window_ms, theta_prefill,
                    theta_decode, dtype="f32", diag=None, stream=None):
    """Stage-aware signal: prefill TSS = (P/dt) / max(A_prefill + w_q W, 1) and
    decode TSS = (D/dt) / max(A_decode, 1), each smoothed and normalised by its
    own theta. Returns (prefill, decode) dicts of S, Z, cls."""
    torch = _torch()
    lib = load()
    K, M = counts["P"].shape
    code, tdt = _dt(dtype)
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    th = [(t if torch.is_tensor(t) else torch.as_tensor(np.asarray(t))).to(
        device="cuda", dtype=tdt).contiguous() for t in (theta_prefill, theta_decode)]
    for t, what in ((A_prefill, "A_prefill"), (A_decode, "A_decode")):
        _need(t, "int32", K * M, what)
    out = [{"S": torch.empty((K, M), dtype=tdt, device="cuda"),
            "Z": torch.empty((K, M), dtype=tdt, device="cuda"),
            "cls": torch.empty((K, M), dtype=torch.uint8, device="cuda")} for _ in range(2)]
    diag = new_diag() if diag is None else diag
    cs = _counts(counts)
    s = _stream(stream)
    _workspace("tss_stage_score", lambda ws, n: lib.tss_stage_score(
        C.byref(g), C.byref(cs), _ptr(A_prefill), _ptr(A_decode), C.byref(pst), _ptr(th[0]),
        _ptr(th[1]), _ptr(out[0]["S"]), _ptr(out[0]["Z"]), _ptr(out[0]["cls"]), _ptr(out[1]["S"]),
        _ptr(out[1]["Z"]), _ptr(out[1]["cls"]), ws, n, _ptr(diag), s))
    return out[0], out[1]


def tss_calibrate(counts, profile, window_ms, slo_ttft_ms, requests=None, events=None,
                  dtype="f32", ok_frac=0.95, reliability=0.95, diag=None, stream=None,
                  S_out=None, cls_out=None):
    """theta per model (CUDA tensor of dtype). S_out / cls_out ([K][M] CUDA
    tensors of dtype / uint8), when given, receive the smoothed series and the
    idle classes the boundary was taken from."""
    torch = _torch()
    lib = load()
    K, M = counts["P"].shape
    code, tdt = _dt(dtype)
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    slo = torch.as_tensor(np.asarray(slo_ttft_ms, np.int32)).cuda() \
        if not torch.is_tensor(slo_ttft_ms) else slo_ttft_ms
    theta = torch.empty(M, dtype=tdt, device="cuda")
    diag = new_diag() if diag is None else diag
    rq = requests_struct(requests) if requests is not None else None
    ev = events_struct(events) if events is not None else None
    cs = _counts(counts)
    s = _stream(stream)
    _workspace("tss_calibrate", lambda ws, n: lib.tss_calibrate(
        C.byref(g), C.byref(rq) if rq else None, C.byref(ev) if ev else None, C.byref(cs),
        C.byref(pst), _ptr(slo), C.c_double(ok_frac), C.c_double(reliability), _ptr(theta),
        _ptr(S_out), _ptr(cls_out), ws, n, _ptr(diag), s))
    return theta


def tss_normalize(S, idle_cls, profile, window_ms, recv=True, Z_out=None, cls_out=None,
                  stream=None):
    """Eq. 2 and the regions (and the Eq. 3 receiver) of a smoothed series:
    returns dict Z, cls (and recv), as tss_score does for the same S."""
    torch = _torch()
    lib = load()
    K, M = S.shape
    code, tdt = _dt(S.dtype)
    _need(idle_cls, "uint8", K * M, "idle_cls")
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    Z = torch.empty((K, M), dtype=tdt, device="cuda") if Z_out is None else Z_out
    cls = torch.empty((K, M), dtype=torch.uint8, device="cuda") if cls_out is None else cls_out
    rv = torch.empty(K, dtype=torch.int32, device="cuda") if recv else None
    _check("tss_normalize", lib.tss_normalize(C.byref(g), C.byref(pst), _ptr(S), _ptr(idle_cls),
                                              _ptr(Z), _ptr(cls), _ptr(rv), _stream(stream)))
    return {"Z": Z, "cls": cls, "recv": rv}


def tre_select_moves(Z, cls, profile, window_ms, budget, r0, r_min, footprint, fast_ms=5000,
                     slow_ms=10000, pacing_cap=1, moves_cap=4096, diag=None, stream=None):
    """Open-loop move selection. Returns (moves [n] structured numpy, r_final
    CUDA tensor, n_moves int, diag)."""
    torch = _torch()
    lib = load()
    K, M = Z.shape
    code, tdt = _dt(Z.dtype)
    g = Grid(M, window_ms, K)
    pst, keep = _profile(profile, M, tdt, code)
    dev = lambda a: (a if torch.is_tensor(a) else torch.as_tensor(np.asarray(a, np.int32))).to(
        device="cuda", dtype=torch.int32).contiguous()
    r = dev(r0).clone()
    rmin, fp = dev(r_min), dev(footprint)
    ctrl = Ctrl(int(budget), rmin.data_ptr(), fp.data_ptr(), fast_ms, slow_ms, pacing_cap)
    moves = torch.zeros(max(moves_cap, 1) * MOVE_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    nmv = torch.zeros(1, dtype=torch.int64, device="cuda")
    diag = new_diag() if diag is None else diag
    s = _stream(stream)
    _workspace("tre_select_moves", lambda ws, n: lib.tre_select_moves(
        C.byref(g), _ptr(Z), _ptr(cls), C.byref(pst), C.byref(ctrl), _ptr(r), _ptr(moves),
        C.c_int64(moves_cap), _ptr(nmv), ws, n, _ptr(diag), s))
    n = int(nmv.item())
    mv = np.frombuffer(moves.cpu().numpy().tobytes(), dtype=MOVE_DTYPE)[: min(n, moves_cap)]
    return mv, r, n, diag


class SweepPlan:
    """A tre_sweep call marshalled once: device parameter arrays, output
    buffers, workspace and the C structs are built here, and run() issues the
    one C call on a stream with no further host work. `traces`: list of dicts
    of int32 CUDA tensors (kept referenced by the plan)."""

    def __init__(self, traces, M, duration_ms, window_ms, alpha, tau_crit, pacing_cap, w_p, w_q,
                 tau_surplus, slo_ttft_ms, budget, r0, r_min, footprint, fast_ms=5000,
                 slow_ms=10000, dtype="f32", ok_frac=0.95, reliability=0.95, moves_cap=256,
                 want_counts=False, want_S=False, diag=None, ws=None):
        torch = _torch()
        self.lib = load()
        code, tdt = _dt(dtype)
        win = np.asarray(window_ms, np.int32)
        n_series = len(traces) * len(win)
        self.K = [duration_ms // int(w) for w in win]
        total = sum(self.K[i % len(win)] * M for i in range(n_series))
        n_inst = n_series * len(tau_crit) * len(pacing_cap)
        f = lambda v: torch.as_tensor(np.broadcast_to(np.asarray(v), (M,)).copy()).to(
            device="cuda", dtype=tdt)
        i32 = lambda v: torch.as_tensor(np.asarray(v, np.int32)).cuda()
        k = {"w_p": f(w_p), "w_q": f(w_q), "ts": f(tau_surplus), "slo": i32(slo_ttft_ms),
             "r0": i32(r0), "rmin": i32(r_min), "fp": i32(footprint)}
        out = {"theta": torch.empty((n_series, M), dtype=tdt, device="cuda"),
               "Z": torch.empty(total, dtype=tdt, device="cuda"),
               "cls": torch.empty(total, dtype=torch.uint8, device="cuda"),
               "moves": torch.zeros(n_inst * max(moves_cap, 1) * MOVE_DTYPE.itemsize,
                                    dtype=torch.uint8, device="cuda"),
               "n_moves": torch.zeros(n_inst, dtype=torch.int64, device="cuda"),
               "r_final": torch.empty((n_inst, M), dtype=torch.int32, device="cuda")}
        if want_counts:
            for c in "PDAW":
                out[c] = torch.empty(total, dtype=torch.int32, device="cuda")
        if want_S:
            out["S"] = torch.empty(total, dtype=tdt, device="cuda")
        self._tr = (Requests * len(traces))(*[requests_struct(t) for t in traces])
        self._wins = (C.c_int32 * len(win))(*[int(x) for x in win])
        self._alph = (C.c_double * len(win))(*[float(a) for a in alpha])
        self._taus = (C.c_double * len(tau_crit))(*[float(t) for t in tau_crit])
        self._caps = (C.c_int32 * len(pacing_cap))(*[int(c) for c in pacing_cap])
        ctrl = Ctrl(int(budget), k["rmin"].data_ptr(), k["fp"].data_ptr(), fast_ms, slow_ms, 0)
        self.spec = SweepSpec(M, duration_ms, len(traces), self._tr, len(win), self._wins,
                              self._alph, len(tau_crit), self._taus, len(pacing_cap), self._caps,
                              code, k["w_p"].data_ptr(), k["w_q"].data_ptr(), k["ts"].data_ptr(),
                              k["slo"].data_ptr(), ok_frac, reliability, ctrl, k["r0"].data_ptr())
        self.sout = SweepOut(*[out[c].data_ptr() if c in out else None
                               for c in ("P", "D", "A", "W", "S", "Z", "cls", "theta", "moves")],
                             moves_cap, out["n_moves"].data_ptr(), out["r_final"].data_ptr())
        size = C.c_size_t(0)
        _check("tre_sweep", self.lib.tre_sweep(C.byref(self.spec), C.byref(self.sout), None,
                                               C.byref(size), None, None))
        if ws is None or ws.numel() < size.value:
            ws = torch.empty(max(int(size.value), 256), dtype=torch.uint8, device="cuda")
        self.diag = new_diag() if diag is None else diag
        out.update(ws=ws, diag=self.diag, K=self.K)
        self.out = out
        self._keep = (k, traces)
        self._ws_ptr = C.c_void_p(ws.data_ptr())
        self._ws_n = C.c_size_t(ws.numel())
        self._diag_ptr = C.c_void_p(self.diag.data_ptr())
        self.n_inst, self.moves_cap = n_inst, moves_cap

    def run(self, stream=None):
        """Enqueue the sweep on `stream` (default: current torch stream); returns
        the plan's output dict (the same tensors every call)."""
        _check("tre_sweep", self.lib.tre_sweep(C.byref(self.spec), C.byref(self.sout),
                                               self._ws_ptr, C.byref(self._ws_n), self._diag_ptr,
                                               _stream(stream)))
        return self.out


def tre_sweep(traces, M, duration_ms, window_ms, alpha, tau_crit, pacing_cap, w_p, w_q,
              tau_surplus, slo_ttft_ms, budget, r0, r_min, footprint, fast_ms=5000,
              slow_ms=10000, dtype="f32", ok_frac=0.95, reliability=0.95, moves_cap=256,
              want_counts=False, want_S=False, diag=None, stream=None, ws=None):
    """Batched open-loop sweep, one call. Returns a dict of CUDA tensors (theta,
    Z, cls, moves, n_moves, r_final, ...) plus the workspace `ws` for reuse."""
    plan = SweepPlan(traces, M, duration_ms, window_ms, alpha, tau_crit, pacing_cap, w_p, w_q,
                     tau_surplus, slo_ttft_ms, budget, r0, r_min, footprint, fast_ms, slow_ms,
                     dtype, ok_frac, reliability, moves_cap, want_counts, want_S, diag, ws)
    out = dict(plan.run(stream))
    out["_keep"] = plan
    return out


def sweep_moves(out, n_inst, moves_cap):
    """Host view of the sweep's move lists: list of structured arrays per instance."""
    raw = np.frombuffer(out["moves"].cpu().numpy().tobytes(), dtype=MOVE_DTYPE)
    raw = raw.reshape(n_inst, max(moves_cap, 1))
    n = out["n_moves"].cpu().numpy()
    return [raw[i, : min(int(n[i]), moves_cap)] for i in range(n_inst)]


class PipelinePlan:
    """One trace's whole path marshalled once: tss_window_reduce ->
    tss_calibrate (which also returns the smoothed series) -> tss_normalize ->
    tre_select_moves, on request records or token events (dicts of
    int32/float32/uint8 CUDA tensors). Device parameter arrays, outputs, one
    workspace (sized for the largest of the calls, which run in order on one
    stream) and the C structs are built here; run() resets the controller's
    replicas to r0 and issues the four C calls with no further host work."""

    def __init__(self, M, window_ms, K, profile, slo_ttft_ms, budget, r0, r_min, footprint,
                 requests=None, events=None, dtype="f32", fast_ms=5000, slow_ms=10000,
                 pacing_cap=1, moves_cap=4096, ok_frac=0.95, reliability=0.95, diag=None):
        torch = _torch()
        self.lib = lib = load()
        code, tdt = _dt(dtype)
        self.g = Grid(M, window_ms, K)
        self.rq = requests_struct(requests) if requests is not None else None
        self.ev = events_struct(events) if events is not None else None
        self._inputs = (requests, events)
        c = {k: torch.empty((K, M), dtype=torch.int32, device="cuda") for k in "PDAW"}
        self.cs = _counts(c)
        prof = dict(profile)
        self.theta = torch.empty(M, dtype=tdt, device="cuda")
        prof["theta"] = self.theta
        self.pst, self._prof = _profile(prof, M, tdt, code)
        i32 = lambda a: (a if torch.is_tensor(a) else torch.as_tensor(np.asarray(a, np.int32))).to(
            device="cuda", dtype=torch.int32).contiguous()
        self.slo = i32(slo_ttft_ms)
        self.r0, self.r = i32(r0), i32(r0).clone()
        self._rmin, self._fp = i32(r_min), i32(footprint)
        self.ctrl = Ctrl(int(budget), self._rmin.data_ptr(), self._fp.data_ptr(), fast_ms, slow_ms,
                         pacing_cap)
        self.S = torch.empty((K, M), dtype=tdt, device="cuda")
        self.Z = torch.empty((K, M), dtype=tdt, device="cuda")
        self.cls = torch.empty((K, M), dtype=torch.uint8, device="cuda")
        self.recv = torch.empty(K, dtype=torch.int32, device="cuda")
        self.moves = torch.zeros(max(moves_cap, 1) * MOVE_DTYPE.itemsize, dtype=torch.uint8,
                                 device="cuda")
        self.n_moves = torch.zeros(1, dtype=torch.int64, device="cuda")
        self.moves_cap = moves_cap
        self.diag = new_diag() if diag is None else diag
        self.ok_frac, self.rel = float(ok_frac), float(reliability)
        self.counts = c
        # one workspace for the four calls
        need = 0
        for q in self._calls(None):
            size = C.c_size_t(0)
            _check(q[0], q[1](None, C.byref(size)))
            need = max(need, int(size.value))
        self.ws = torch.empty(max(need, 256), dtype=torch.uint8, device="cuda")
        self._ws_n = C.c_size_t(self.ws.numel())

    def _calls(self, stream):
        lib, g, P = self.lib, self.g, C.c_void_p
        rq = C.byref(self.rq) if self.rq is not None else None
        ev = C.byref(self.ev) if self.ev is not None else None
        dg = _ptr(self.diag)
        return (
            ("tss_window_reduce", lambda ws, n: lib.tss_window_reduce(
                C.byref(g), rq, ev, self.cs, ws, n, dg, stream)),
            ("tss_calibrate", lambda ws, n: lib.tss_calibrate(
                C.byref(g), rq, ev, C.byref(self.cs), C.byref(self.pst), _ptr(self.slo),
                C.c_double(self.ok_frac), C.c_double(self.rel), _ptr(self.theta), _ptr(self.S),
                _ptr(self.cls), ws, n, dg, stream)),
            # Z and regions from the series calibrate smoothed (no workspace)
            ("tss_normalize", lambda ws, n: lib.tss_normalize(
                C.byref(g), C.byref(self.pst), _ptr(self.S), _ptr(self.cls), _ptr(self.Z),
                _ptr(self.cls), _ptr(self.recv), stream) if ws is not None else 0),
            ("tre_select_moves", lambda ws, n: lib.tre_select_moves(
                C.byref(g), _ptr(self.Z), _ptr(self.cls), C.byref(self.pst), C.byref(self.ctrl),
                _ptr(self.r), _ptr(self.moves), C.c_int64(self.moves_cap), _ptr(self.n_moves),
                ws, n, dg, stream)),
        )

    def run(self, stream=None):
        """Enqueue the whole path on `stream` (default: current torch stream)."""
        torch = _torch()
        s = stream if stream is not None else torch.cuda.current_stream()
        with torch.cuda.stream(s):
            self.r.copy_(self.r0, non_blocking=True)
        ws = C.c_void_p(self.ws.data_ptr())
        for name, fn in self._calls(C.c_void_p(s.cuda_stream)):
            _check(name, fn(ws, C.byref(self._ws_n)))
        return self

    def results(self):
        """Host view of the last run: counts, theta, S, Z, cls, recv, moves, r_final."""
        n = int(self.n_moves.item())
        mv = np.frombuffer(self.moves.cpu().numpy().tobytes(),
                           dtype=MOVE_DTYPE)[: min(n, self.moves_cap)]
        out = {k: v.cpu().numpy() for k, v in self.counts.items()}
        out.update(theta=self.theta.cpu().numpy(), S=self.S.cpu().numpy(), Z=self.Z.cpu().numpy(),
                   cls=self.cls.cpu().numpy(), recv=self.recv.cpu().numpy(), moves=mv,
                   n_moves=n, r_final=self.r.cpu().numpy())
        return out


LATENT_KEYS = ("model", "t_arr_ms", "d_first_ms", "d_total_ms", "L_in", "L_out")


class ReplayPlan:
    """A tre_replay call marshalled once: the closed-loop replay of one latent
    trace (dict of int32 CUDA tensors, LATENT_KEYS) for every (rescue
    threshold, pacing cap) setting. tau_list None: the profile's tau_crit;
    cap_list None: pacing_cap. guard_ttft_ms: per-model latency guard (None:
    no guard). records / signal: also return the served records and the Z /
    class rows each instance saw. run() issues the call."""

    def __init__(self, latent, M, window_ms, K, profile, budget, r0, r_min, footprint,
                 fast_ms=5000, slow_ms=10000, pacing_cap=1, tau_list=None, cap_list=None,
                 wake_ms=0, sleep_ms=0, slo_ttft_ms=None, guard_ttft_ms=None, dtype="f64",
                 records=False, signal=False, moves_cap=4096, diag=None):
        torch = _torch()
        self.lib = lib = load()
        code, tdt = _dt(dtype)
        n = int(latent["model"].numel())
        for k in LATENT_KEYS:
            _need(latent[k], "int32", n, k)
        self._lat = latent
        self.lat = Latent(n, *[latent[k].data_ptr() if n else None for k in LATENT_KEYS])
        self.g = Grid(M, window_ms, K)
        self.pst, self._prof = _profile(profile, M, tdt, code)
        i32 = lambda a: (a if torch.is_tensor(a) else torch.as_tensor(np.asarray(a, np.int32))).to(
            device="cuda", dtype=torch.int32).contiguous()
        self._r0, self._rmin, self._fp = i32(r0), i32(r_min), i32(footprint)
        self.ctrl = Ctrl(int(budget), self._rmin.data_ptr(), self._fp.data_ptr(), fast_ms, slow_ms,
                         pacing_cap)
        taus = [] if tau_list is None else [float(t) for t in tau_list]
        caps = [] if cap_list is None else [int(c) for c in cap_list]
        self._taus = (C.c_double * max(len(taus), 1))(*taus)
        self._caps = (C.c_int32 * max(len(caps), 1))(*caps)
        self._guard = i32(guard_ttft_ms) if guard_ttft_ms is not None else None
        self.spec = ReplaySpec(len(taus), self._taus, len(caps), self._caps, wake_ms, sleep_ms,
                               self._guard.data_ptr() if self._guard is not None else None)
        self.n_inst = max(len(taus), 1) * max(len(caps), 1)
        ni = self.n_inst
        self.slo = i32(slo_ttft_ms) if slo_ttft_ms is not None else None
        o = {"moves": torch.zeros(ni * max(moves_cap, 1) * MOVE_DTYPE.itemsize, dtype=torch.uint8,
                                  device="cuda"),
             "n_moves": torch.zeros(ni, dtype=torch.int64, device="cuda"),
             "r_final": torch.zeros((ni, M), dtype=torch.int32, device="cuda"),
             "served": torch.zeros((ni, M), dtype=torch.int64, device="cuda")}
        if self.slo is not None:
            o["slo_met"] = torch.zeros((ni, M), dtype=torch.int64, device="cuda")
        if records:
            for k in ("t_start_ms", "t_first_ms", "t_end_ms"):
                o[k] = torch.empty((ni, n), dtype=torch.int32, device="cuda")
        if signal:
            o["Z"] = torch.empty((ni, K, M), dtype=tdt, device="cuda")
            o["cls"] = torch.empty((ni, K, M), dtype=torch.uint8, device="cuda")
        self.out = o
        self.moves_cap = moves_cap
        self.sout = ReplayOut(*[o[k].data_ptr() if k in o else None
                                for k in ("t_start_ms", "t_first_ms", "t_end_ms", "Z", "cls",
                                          "moves")],
                              moves_cap, o["n_moves"].data_ptr(), o["r_final"].data_ptr(),
                              o["slo_met"].data_ptr() if "slo_met" in o else None,
                              o["served"].data_ptr())
        self.diag = new_diag() if diag is None else diag
        size = C.c_size_t(0)
        _check("tre_replay", self._call(None, size, None))
        self.ws = torch.empty(max(int(size.value), 256), dtype=torch.uint8, device="cuda")
        self._ws_n = C.c_size_t(self.ws.numel())

    def _call(self, ws, size, stream):
        return self.lib.tre_replay(C.byref(self.g), C.byref(self.lat), C.byref(self.pst),
                                   C.byref(self.ctrl), _ptr(self._r0), C.byref(self.spec),
                                   _ptr(self.slo), C.byref(self.sout), ws, C.byref(size),
                                   _ptr(self.diag), stream)

    def run(self, stream=None):
        """Enqueue the replay on `stream` (default: current torch stream)."""
        _check("tre_replay", self._call(C.c_void_p(self.ws.data_ptr()), self._ws_n,
                                        _stream(stream)))
        return self.out

    def moves(self):
        """Host view of the move lists: one structured array per instance."""
        raw = np.frombuffer(self.out["moves"].cpu().numpy().tobytes(), dtype=MOVE_DTYPE)
        raw = raw.reshape(self.n_inst, max(self.moves_cap, 1))
        n = self.out["n_moves"].cpu().numpy()
        return [raw[i, : min(int(n[i]), self.moves_cap)] for i in range(self.n_inst)]


def tre_replay(latent, M, window_ms, K, profile, budget, r0, r_min, footprint, **kw):
    """Closed-loop replay, one call (see ReplayPlan). Returns (outputs dict of
    CUDA tensors, list of host move arrays per instance, diag)."""
    plan = ReplayPlan(latent, M, window_ms, K, profile, budget, r0, r_min, footprint, **kw)
    out = plan.run()
    return out, plan.moves(), plan.diag
