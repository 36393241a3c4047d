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
    occ = [cnt_dev[k].data_ptr() if cnt_dev.get(k) is not None else None
           for k in ("A_ms", "W_ms")]
    cs = tre.Counts(*[cnt_dev[k].data_ptr() for k in "PDAW"], *occ)
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


def _profile(rng, M, win):
    return {"w_p": rng.uniform(0.1, 0.3, M), "w_q": rng.uniform(1, 3, M),
            "alpha": np.full(M, min(1.0, win / 5000)), "theta": rng.uniform(5, 50, M),
            "tau_crit": np.full(M, 0.8), "tau_surplus": np.full(M, 1.2)}


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_noalloc_time_averaged_occupancy_matches_tss_score_twice(dtype):
    """The window-mean running and waiting counts (A_ms, W_ms) take their own
    scoring branch; the no-workspace call must follow it exactly too."""
    import torch
    import paper_2609_29160_gb300 as tre
    lib = tre.load()
    lib.tss_score_noalloc.restype = C.c_int
    K, M, win = 9000, 8, 100
    rng = np.random.default_rng(17)
    host = _case(rng, K, M)
    host["A_ms"] = (host["A"].astype(np.int64) * win - rng.integers(0, win, (K, M)) *
                    (host["A"] > 0)).astype(np.int64)
    host["W_ms"] = (host["W"].astype(np.int64) * rng.integers(0, win + 1, (K, M))).astype(np.int64)
    cnt = {k: torch.as_tensor(v).cuda() for k, v in host.items()}
    tdt = torch.float32 if dtype == "f32" else torch.float64
    prof = _profile(rng, M, win)
    ref = tre.tss_score(cnt, prof, win, dtype=dtype)
    prof_st, keep = tre._profile(prof, M, tdt, tre.F32 if dtype == "f32" else tre.F64)
    for _ in range(2):
        got = _call_noalloc(tre, lib, cnt, prof_st, K, M, win, tdt)
        torch.cuda.synchronize()
        for k in ("S", "Z", "cls", "recv"):
            assert torch.equal(got[k], ref[k]), k


@pytest.mark.parametrize("dtype", ["f32", "f64"])
def test_noalloc_carries_smoothing_across_calls(dtype):
    """Two consecutive window ranges scored with the smoothing state carried
    from the first call into the second give what tss_score gives with the
    same carries."""
    import torch
    import paper_2609_29160_gb300 as tre
    lib = tre.load()
    lib.tss_score_noalloc.restype = C.c_int
    K, M, win = 12000, 5, 500
    rng = np.random.default_rng(23)
    host = _case(rng, K, M)
    host["P"][:3000, 1] = 0
    host["D"][:3000, 1] = 0
    host["A"][:3000, 1] = 0
    host["W"][:3000, 1] = 0            # model 1 still uninitialised at the split
    tdt = torch.float32 if dtype == "f32" else torch.float64
    prof = _profile(rng, M, win)
    prof_st, keep = tre._profile(prof, M, tdt, tre.F32 if dtype == "f32" else tre.F64)
    cut = 2500
    halves = [{k: torch.as_tensor(np.ascontiguousarray(v[:cut])).cuda() for k, v in host.items()},
              {k: torch.as_tensor(np.ascontiguousarray(v[cut:])).cuda() for k, v in host.items()}]
    ref_c = {"S": torch.zeros(M, dtype=tdt, device="cuda"),
             "init": torch.zeros(M, dtype=torch.uint8, device="cuda")}
    got_c = {"S": torch.zeros(M, dtype=tdt, device="cuda"),
             "init": torch.zeros(M, dtype=torch.uint8, device="cuda")}
    for h in halves:
        Kh = int(h["P"].shape[0])
        ref = tre.tss_score(h, prof, win, dtype=dtype, carry=ref_c)
        got = _call_noalloc(tre, lib, h, prof_st, Kh, M, win, tdt, carry=got_c)
        torch.cuda.synchronize()
        for k in ("S", "Z", "cls", "recv"):
            assert torch.equal(got[k], ref[k]), k
        assert torch.equal(got_c["S"], ref_c["S"]) and torch.equal(got_c["init"], ref_c["init"])
    assert int(got_c["init"].sum()) == M


def test_noalloc_refuses_one_occupancy_array_without_the_other():
    import paper_2609_29160_gb300 as tre
    lib = tre.load()
    lib.tss_score_noalloc.restype = C.c_int
    g = tre.Grid(4, 100, 10)
    cs = tre.Counts(8, 8, 8, 8, 8, None)
    prof = tre.Profile(0, 8, 8, 8, 8, 8, 8)
    st = lib.tss_score_noalloc(C.byref(g), C.byref(cs), C.byref(prof), None, None,
                               C.c_void_p(8), C.c_void_p(8), C.c_void_p(8), None, C.c_void_p(8),
                               None)
    assert st == 1          # TRE_EINVAL, as tss_score returns
