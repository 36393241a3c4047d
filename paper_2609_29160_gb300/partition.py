"""Splitting the path over several GPUs (one process per GPU).

Two partitions, both exact:

* the open-loop sweep: its traces are independent problems, so rank r takes
  the traces t with t % n_ranks == r and runs tre_sweep on them alone; no data
  moves between ranks;
* one long trace (the 64-model token stream): reduction, smoothing,
  calibration and scoring are independent per model (Eq. 1 and the smoothing
  of Sec. III-B read one model's telemetry; theta is a per-model statistic), so
  rank r takes a contiguous block of models -- its events or records, with
  model ids and request ids renumbered locally -- and runs the per-trace path
  on them. The controller's walk (Sec. IV-B/IV-C) reads every model's Z and
  region at control ticks only: the exchange step gathers those tick rows
  from all ranks (one all-gather of n_ticks x n_models values), after which
  the walk runs on a series with one window per fast tick (the fast cadence as
  its window length), which makes the same decisions as the walk over every
  window.

This module holds the host-side plumbing only (index bookkeeping and the
collective); every step of the computation runs in libtre.so.
"""
from __future__ import annotations

import numpy as np


def sweep_traces(n_traces, rank, n_ranks):
    """Trace indices of rank `rank`: t with t % n_ranks == rank."""
    return [t for t in range(n_traces) if t % n_ranks == rank]


def model_blocks(M, n_ranks):
    """Contiguous model blocks [(m0, m1)] for the ranks, sizes differing by at
    most one (a rank may get none when there are more ranks than models)."""
    base, extra = divmod(M, n_ranks)
    out, m0 = [], 0
    for r in range(n_ranks):
        m1 = m0 + base + (1 if r < extra else 0)
        out.append((m0, m1))
        m0 = m1
    return out


def requests_for_models(req, m0, m1):
    """The request records of models [m0, m1), model ids made local (m - m0).
    Records with a model id outside [0, M) belong to no block; they are
    dropped by every rank (the unsplit reduction counts them as bad ids)."""
    keep = (req["model"] >= m0) & (req["model"] < m1)
    out = {k: np.ascontiguousarray(v[keep]) for k, v in req.items()}
    out["model"] = (out["model"] - m0).astype(np.int32)
    return out


def events_for_models(ev, m0, m1):
    """The token events of models [m0, m1) and their requests' table, with
    model ids local (m - m0) and request ids renumbered into the local table.
    An event whose request id is outside the table, or whose model does not
    match its request's, keeps a local request id the library rejects (-1),
    as the unsplit reduction rejects it."""
    rm = ev["req_model"]
    rows = np.flatnonzero((rm >= m0) & (rm < m1))
    local_id = np.full(len(rm), -1, np.int64)
    local_id[rows] = np.arange(len(rows))
    keep = (ev["model"] >= m0) & (ev["model"] < m1)
    req = ev["req"][keep].astype(np.int64)
    inside = (req >= 0) & (req < len(rm))
    lreq = np.where(inside, local_id[np.clip(req, 0, len(rm) - 1)], -1)
    return {"model": (ev["model"][keep] - m0).astype(np.int32),
            "req": lreq.astype(np.int32),
            "t_s": np.ascontiguousarray(ev["t_s"][keep]),
            "phase": np.ascontiguousarray(ev["phase"][keep]),
            "req_model": (rm[rows] - m0).astype(np.int32),
            "req_t_arr_ms": np.ascontiguousarray(ev["req_t_arr_ms"][rows]),
            "req_ttft_ms": np.ascontiguousarray(ev["req_ttft_ms"][rows])}


def tick_windows(K, window_ms, fast_ms, slow_ms):
    """Windows that end a fast tick, when the cadences nest (window length
    divides the fast cadence, which divides the slow one): then every slow tick
    is a fast tick and the walk reads nothing else."""
    if fast_ms % window_ms or slow_ms % fast_ms:
        raise ValueError("tick rows need window_ms | fast_ms | slow_ms")
    q = fast_ms // window_ms
    return np.arange(q - 1, K, q, dtype=np.int64)


def moves_to_windows(moves, window_ms, fast_ms):
    """Map the windows of moves made on the tick series (one window per fast
    tick) back to the original windows."""
    out = moves.copy()
    q = fast_ms // window_ms
    out["window"] = (out["window"].astype(np.int64) * q + q - 1).astype(out["window"].dtype)
    return out


def gather_tick_rows(dist, Z_ticks, cls_ticks, blocks, group=None):
    """The exchange step: every rank contributes its models' Z and region rows
    at the tick windows ([n_ticks][m1 - m0] tensors, same dtype and device on
    every rank); returns the full [n_ticks][M] rows on every rank. Blocks may
    differ in width by one, so rows are padded to the widest block for the
    all-gather and cut back after it."""
    import torch
    n_ticks = Z_ticks.shape[0]
    width = max(m1 - m0 for m0, m1 in blocks)
    M = blocks[-1][1]
    zp = torch.zeros((n_ticks, width), dtype=Z_ticks.dtype, device=Z_ticks.device)
    cp = torch.zeros((n_ticks, width), dtype=torch.int32, device=Z_ticks.device)
    zp[:, :Z_ticks.shape[1]] = Z_ticks
    cp[:, :cls_ticks.shape[1]] = cls_ticks.to(torch.int32)
    zs = [torch.empty_like(zp) for _ in blocks]
    cs = [torch.empty_like(cp) for _ in blocks]
    dist.all_gather(zs, zp, group=group)
    dist.all_gather(cs, cp, group=group)
    Z = torch.empty((n_ticks, M), dtype=Z_ticks.dtype, device=Z_ticks.device)
    cls = torch.empty((n_ticks, M), dtype=torch.uint8, device=Z_ticks.device)
    for (m0, m1), z, c in zip(blocks, zs, cs):
        Z[:, m0:m1] = z[:, : m1 - m0]
        cls[:, m0:m1] = c[:, : m1 - m0].to(torch.uint8)
    return Z, cls


def block_signal(tre, block, window_ms, K, profile, slo_ttft_ms, dtype="f32", stream=None):
    """One rank's share of a long trace through the library: counts, theta,
    and Z / regions of its models. `block`: the rank's telemetry as CUDA
    tensors, {"requests": {...}} or {"events": {...}}, with local ids; the
    profile and SLO bounds are the block's models' ([m1 - m0])."""
    M = int(len(slo_ttft_ms))
    kw = {k: v for k, v in block.items()}
    import torch
    c = tre.tss_window_reduce(M, window_ms, K, stream=stream, **kw)
    S = torch.empty((K, M), dtype=torch.float32 if dtype == "f32" else torch.float64,
                    device="cuda")
    cls = torch.empty((K, M), dtype=torch.uint8, device="cuda")
    theta = tre.tss_calibrate(c, profile, window_ms, slo_ttft_ms, dtype=dtype, stream=stream,
                              S_out=S, cls_out=cls, **kw)
    sc = tre.tss_normalize(S, cls, dict(profile, theta=theta), window_ms, recv=False,
                           cls_out=cls, stream=stream)
    return {"counts": c, "theta": theta, "Z": sc["Z"], "cls": sc["cls"], "S": S}


def walk_on_ticks(tre, Z_ticks, cls_ticks, profile, window_ms, fast_ms, slow_ms, budget, r0,
                  r_min, footprint, pacing_cap=1, moves_cap=1 << 16, stream=None):
    """The controller's walk over gathered tick rows (one window per fast tick,
    the fast cadence as window length); moves come back on the original
    windows."""
    mv, r, n, diag = tre.tre_select_moves(Z_ticks.contiguous(), cls_ticks.contiguous(), profile,
                                          fast_ms, budget, r0, r_min, footprint,
                                          fast_ms=fast_ms, slow_ms=slow_ms,
                                          pacing_cap=pacing_cap, moves_cap=moves_cap,
                                          stream=stream)
    return moves_to_windows(mv, window_ms, fast_ms), r, n, diag
