"""tss_score_noalloc: scoring for callers that cannot allocate device memory and
so cannot hand the library a workspace. Called through the C ABI, it must give
exactly what tss_score gives -- on two calls in a row, since every call reuses
the same built-in scratch buffer -- and refuse problems larger than that
buffer before touching the device."""
import ctypes as C

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def _case(rng, K, M):
    cnt = {k: rng.integers(0, hi, (K, M)).astype(np.int32)
           for k, hi in (("P", 4000), ("D", 700), ("A", 25), ("W", 50))}
    idle = rng.random((K, M)) < 0.2
    for v in cnt.values():
        v[idle] = 0
    return cnt


def _call_noalloc(tre, lib, cnt_dev, prof_st, K, M, win, tdt, carry=None):
    import torch
    S = torch.empty((K, M), dtype=tdt, device="cuda")
    Z = torch.empty((K, M), dtype=tdt, device="cuda")
    cls = torch.empty((K, M), dtype=torch.uint8, device="cuda")
    recv = torch.empty(K, dtype=torch.int32, device="cuda")
    diag = tre.new_diag()
    g = tre.Grid(M, win, K)
    cs = tre.Counts(*[cnt_dev[k].data_ptr() for k in "PDAW"])
    st = lib.tss_score_noalloc(C.byref(g), C.byref(cs), C.byref(prof_st),
                               C.c_void_p(carry["S"].data_ptr()) if carry else None,
                               C.c_void_p(carry["init"].data_ptr()) if carry else None,
                               C.c_void_p(S.data_ptr()), C.c_void_p(Z.data_ptr()),
                               C.c_void_p(cls.data_ptr()), C.c_void_p(recv.data_ptr()),
                               C.c_void_p(diag.data_ptr()),
                               C.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 0, st
    return {"S": S, "Z": Z, "cls": cls, "recv": recv}


@pytest.mark.parametrize("dtype", ["f32", "f64"])
@pytest.mark.parametrize("K,M,win", [(36000, 8, 100), (600, 3, 1000), (16384, 64, 100)])
def test_noalloc_matches_tss_score_twice(dtype, K, M, win):
    import torch
    import paper_2609_29160_gb300 as tre
    lib = tre.load()
    lib.tss_score_noalloc.restype = C.c_int
    rng = np.random.default_rng(K + M)
    cnt = {k: torch.as_tensor(v).cuda() for k, v in _case(rng, K, M).items()}
    tdt = torch.float32 if dtype == "f32" else torch.float64
    prof = {"w_p": rng.uniform(0.1, 0.3, M), "w_q": rng.uniform(1, 3, M),
            "alpha": np.full(M, min(1.0, win / 5000)), "theta": rng.uniform(5, 50, M),
            "tau_crit": np.full(M, 0.8), "tau_surplus": np.full(M, 1.2)}
    ref = tre.tss_score(cnt, prof, win, dtype=dtype)
    prof_st, keep = tre._profile(prof, M, tdt, tre.F32 if dtype == "f32" else tre.F64)
    for _ in range(2):
        got = _call_noalloc(tre, lib, cnt, prof_st, K, M, win, tdt)
        torch.cuda.synchronize()
        for k in ("S", "Z", "cls", "recv"):
            assert torch.equal(got[k], ref[k]), k


def test_noalloc_rejects_problems_beyond_its_buffer():
    import paper_2609_29160_gb300 as tre
    lib = tre.load()
    lib.tss_score_noalloc.restype = C.c_int
    g = tre.Grid(64, 100, 16385)        # 16385 x 64 cells > 2^20
    cs = tre.Counts(8, 8, 8, 8)
    prof = tre.Profile(0, 8, 8, 8, 8, 8, 8)
    st = lib.tss_score_noalloc(C.byref(g), C.byref(cs), C.byref(prof), None, None,
                               C.c_void_p(8), C.c_void_p(8), C.c_void_p(8), None, C.c_void_p(8),
                               None)
    assert st == 2          # TRE_ENOMEM, nothing enqueued
