"""The C-ABI library builds for sm_103a, loads, and exports every entry point
that include/tre.h declares; host-side argument checks answer without a GPU
(no compute call is made here)."""
import ctypes as C
import os
import re

import pytest

import paper_2609_29160_gb300 as tre
from tests.conftest import ROOT


def _declared():
    src = open(os.path.join(ROOT, "include", "tre.h")).read()
    return sorted(set(re.findall(r"^(?:tre_status|const char\*)\s+(\w+)\s*\(", src, re.M)))


def test_header_declares_the_five_entry_points():
    names = _declared()
    for n in ("tss_window_reduce", "tss_score", "tss_calibrate", "tre_select_moves", "tre_sweep",
              "tre_status_str"):
        assert n in names


def test_library_exports_every_declared_symbol():
    lib = tre.load()
    for name in _declared():
        assert hasattr(lib, name), name


def test_struct_layouts_match_header_sizes():
    # sizes fixed by the header's field lists on LP64
    assert C.sizeof(tre.Grid) == 12
    assert C.sizeof(tre.Requests) == 8 + 7 * 8
    assert C.sizeof(tre.Diag) == 5 * 8 + 8
    assert tre.MOVE_DTYPE.itemsize == 12


def test_status_strings():
    lib = tre.load()
    assert lib.tre_status_str(0) == b"ok"
    assert lib.tre_status_str(4) == b"move list overflow"


def test_argument_errors_are_reported_on_the_host():
    lib = tre.load()
    g = tre.Grid(0, 1000, 10)           # no models
    n = C.c_size_t(0)
    rq = tre.Requests(0)
    cs = tre.Counts(1, 1, 1, 1)
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq), None, cs, None, C.byref(n), None,
                                 None) == 1
    g = tre.Grid(3, 1000, 10)
    # both and neither telemetry descriptor
    ev = tre.Events(0)
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq), C.byref(ev), cs, None, C.byref(n),
                                 None, None) == 1
    assert lib.tss_window_reduce(C.byref(g), None, None, cs, None, C.byref(n), None, None) == 1
    # a workspace query needs no device
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq), None, cs, None, C.byref(n), None,
                                 None) == 0
    assert n.value > 0
    # records present but a column missing
    rq2 = tre.Requests(5, 1, 1, 1, 1, 1, 1, None)
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq2), None, cs, None, C.byref(n), None,
                                 None) == 1
    # window grid beyond int32 milliseconds
    big = tre.Grid(3, 1_000_000, 10_000)
    assert lib.tss_window_reduce(C.byref(big), C.byref(rq), None, cs, None, C.byref(n), None,
                                 None) == 1


def test_workspace_too_small_is_enomem():
    lib = tre.load()
    g = tre.Grid(4, 100, 1000)
    cs = tre.Counts(1, 1, 1, 1)
    prof = tre.Profile(0, 8, 8, 8, 8, 8, 8)
    n = C.c_size_t(0)
    assert lib.tss_score(C.byref(g), C.byref(cs), C.byref(prof), None, None, 8, 8, 8, None, None,
                         C.byref(n), None, None) == 0
    need = n.value
    small = C.c_size_t(need - 1)
    assert lib.tss_score(C.byref(g), C.byref(cs), C.byref(prof), None, None, 8, 8, 8, None,
                         C.c_void_p(4096), C.byref(small), C.c_void_p(8), None) == 2


def test_select_and_sweep_argument_checks():
    lib = tre.load()
    g = tre.Grid(3, 1000, 100)
    prof = tre.Profile(0, 8, 8, 8, 8, 8, 8)
    n = C.c_size_t(0)
    bad = tre.Ctrl(8, 8, 8, 5000, 10000, 300)     # pacing cap beyond one byte of seq
    assert lib.tre_select_moves(C.byref(g), 8, 8, C.byref(prof), C.byref(bad), 8, 8, 10, 8, None,
                                C.byref(n), None, None) == 1
    ok = tre.Ctrl(8, 8, 8, 5000, 10000, 1)
    assert lib.tre_select_moves(C.byref(g), 8, 8, C.byref(prof), C.byref(ok), 8, 8, 10, 8, None,
                                C.byref(n), None, None) == 0
    # sweep window lengths that do not nest
    tr = (tre.Requests * 1)(tre.Requests(0))
    wins = (C.c_int32 * 2)(300, 500)
    al = (C.c_double * 2)(0.1, 0.1)
    tau = (C.c_double * 1)(0.8)
    cap = (C.c_int32 * 1)(1)
    spec = tre.SweepSpec(3, 3000, 1, tr, 2, wins, al, 1, tau, 1, cap, 0, 8, 8, 8, 8, 0.95, 0.95,
                         tre.Ctrl(8, 8, 8, 5000, 10000, 0), 8)
    so = tre.SweepOut(None, None, None, None, None, None, None, 8, 8, 4, 8, 8)
    assert lib.tre_sweep(C.byref(spec), C.byref(so), None, C.byref(n), None, None) == 1
    wins2 = (C.c_int32 * 2)(500, 1000)
    spec.window_ms = wins2
    assert lib.tre_sweep(C.byref(spec), C.byref(so), None, C.byref(n), None, None) == 0


def test_rank_argument_errors_are_reported_on_the_host():
    lib = tre.load()
    g = tre.Grid(4, 1000, 10)
    out = C.c_void_p(16)        # never dereferenced: the checks fail first
    assert lib.tss_rank(C.byref(g), 2, out, out, out, None, None) == 1    # unknown dtype
    assert lib.tss_rank(C.byref(g), 0, None, out, out, None, None) == 1   # Z missing
    assert lib.tss_rank(C.byref(g), 1, out, None, None, out, None) == 1   # cls missing
    assert lib.tss_rank(None, 0, out, out, out, None, None) == 1
    g0 = tre.Grid(4, 1000, 0)   # empty grid: nothing to enqueue
    assert lib.tss_rank(C.byref(g0), 0, None, None, out, out, None) == 0


def test_mean_occupancy_arguments_are_checked_on_the_host():
    lib = tre.load()
    g = tre.Grid(3, 1000, 10)
    n = C.c_size_t(0)
    rq = tre.Requests(0)
    ev = tre.Events(0)
    one_sided = tre.Counts(1, 1, 1, 1, 1, None)          # A_ms without W_ms
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq), None, one_sided, None, C.byref(n),
                                 None, None) == 1
    both = tre.Counts(1, 1, 1, 1, 1, 1)
    assert lib.tss_window_reduce(C.byref(g), None, C.byref(ev), both, None, C.byref(n), None,
                                 None) == 0              # token events: workspace query
    assert lib.tss_window_reduce(C.byref(g), C.byref(rq), None, both, None, C.byref(n), None,
                                 None) == 0              # workspace query


def test_class_models_arguments_are_checked_on_the_host():
    lib = tre.load()
    p = C.c_void_p(16)          # never dereferenced: the checks fail first
    assert lib.tss_class_models(10, p, p, 0, 3, p, None) == 1      # no models
    assert lib.tss_class_models(10, p, p, 8, 0, p, None) == 1      # no classes
    assert lib.tss_class_models(10, p, p, 400, 3, p, None) == 1    # more than 1024 pairs
    assert lib.tss_class_models(10, None, p, 8, 3, p, None) == 1
    assert lib.tss_class_models(0, None, None, 8, 3, None, None) == 0


def test_binding_checks_tensor_arguments():
    import torch
    keys = ("model", "t_arr_ms", "t_start_ms", "t_first_ms", "t_end_ms", "L_in", "L_out")
    good = {k: torch.zeros(5, dtype=torch.int32) for k in keys}
    assert tre.requests_struct(good).n == 5
    with pytest.raises(ValueError, match="int32"):
        tre.requests_struct(dict(good, L_out=torch.zeros(5, dtype=torch.int64)))
    with pytest.raises(ValueError, match="elements"):
        tre.requests_struct(dict(good, t_end_ms=torch.zeros(4, dtype=torch.int32)))
    with pytest.raises(ValueError, match="contiguous"):
        tre.requests_struct(dict(good, t_arr_ms=torch.zeros(10, dtype=torch.int32)[::2]))
    cnt = {k: torch.zeros((3, 2), dtype=torch.int32) for k in "PDAW"}
    tre._counts(cnt)
    with pytest.raises(ValueError, match="int64"):
        tre._counts(dict(cnt, A_ms=torch.zeros((3, 2), dtype=torch.int32),
                         W_ms=torch.zeros((3, 2), dtype=torch.int64)))



def test_stage_arguments_are_checked_on_the_host():
    lib = tre.load()
    g = tre.Grid(3, 1000, 10)
    n = C.c_size_t(0)
    rq = tre.Requests(0)
    p = C.c_void_p(16)          # never dereferenced: the checks fail first
    assert lib.tss_stage_gauges(C.byref(g), C.byref(rq), p, None, None, C.byref(n), None,
                                None) == 1              # A_decode missing
    assert lib.tss_stage_gauges(C.byref(g), C.byref(rq), p, p, None, C.byref(n), None,
                                None) == 0              # workspace query
    cs = tre.Counts(16, 16, 16, 16, 16, 16)             # window means: not for stages
    prof = tre.Profile(0, 16, 16, 16, 16, 16, 16)
    assert lib.tss_stage_score(C.byref(g), C.byref(cs), p, p, C.byref(prof), p, p, p, p, p, p,
                               p, p, None, C.byref(n), None, None) == 1
    cs = tre.Counts(16, 16, 16, 16)
    assert lib.tss_stage_score(C.byref(g), C.byref(cs), p, p, C.byref(prof), p, p, p, p, p, p,
                               p, p, None, C.byref(n), None, None) == 0
    assert lib.tss_stage_calibrate(C.byref(g), C.byref(rq), C.byref(cs), p, p, C.byref(prof), p,
                                   None, 0.95, 0.95, p, p, None, C.byref(n), None,
                                   None) == 1           # TPOT bounds missing
    assert lib.tss_stage_calibrate(C.byref(g), C.byref(rq), C.byref(cs), p, p, C.byref(prof), p,
                                   p, 0.95, 0.95, p, p, None, C.byref(n), None, None) == 0


def test_normalize_argument_checks():
    """tss_normalize refuses a profile without theta or thresholds and missing
    arrays, and an empty grid is a no-op; none of these touches the device."""
    lib = tre.load()
    g = tre.Grid(4, 100, 1000)
    full = tre.Profile(0, 8, 8, 8, 8, 8, 8)
    no_theta = tre.Profile(0, 8, 8, 8, None, 8, 8)
    assert lib.tss_normalize(C.byref(g), C.byref(no_theta), 8, 8, 8, 8, None, None) == 1
    assert lib.tss_normalize(C.byref(g), C.byref(full), None, 8, 8, 8, None, None) == 1
    assert lib.tss_normalize(C.byref(g), C.byref(full), 8, 8, 8, None, None, None) == 1
    bad_dtype = tre.Profile(7, 8, 8, 8, 8, 8, 8)
    assert lib.tss_normalize(C.byref(g), C.byref(bad_dtype), 8, 8, 8, 8, None, None) == 1
    empty = tre.Grid(4, 100, 0)
    assert lib.tss_normalize(C.byref(empty), C.byref(full), None, None, None, None, None,
                             None) == 0
