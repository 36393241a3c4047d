"""The multi-GPU partitions run as shards in sequence on one GPU, through the
library, against the unsplit call, bit for bit:

* a 64-model token stream split into model blocks: each block's counts,
  theta, Z and regions equal the unsplit columns, and the walk over the
  blocks' tick rows put side by side (what the all-gather delivers) makes the
  unsplit moves and final replicas;
* the open-loop sweep split by traces: each shard's series and controller
  instances equal the corresponding ones of the whole sweep."""
import numpy as np
import pytest

import tracegen

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def tre():
    import torch
    import paper_2609_29160_gb300 as lib
    lib.load()
    torch.cuda.set_device(0)
    return lib


def _cuda(d):
    import torch
    return {k: torch.as_tensor(np.ascontiguousarray(v)).cuda() for k, v in d.items()}


@pytest.mark.parametrize("n_shards", [2, 5, 8])
def test_model_blocks_of_a_token_stream(tre, n_shards):
    import torch
    from paper_2609_29160_gb300 import partition
    w = tracegen.workload("stream", scale=0.02)
    M, win, K = w["M"], w["window_ms"], w["K"]
    prof = tracegen.default_profile(M, win)
    plan = tre.PipelinePlan(M, win, K, prof, w["slo_ttft_ms"], w["budget"], w["r0"], w["r_min"],
                            w["footprint"], events=_cuda(w["events"]), moves_cap=1 << 16)
    plan.run()
    ref = plan.results()
    assert ref["n_moves"] > 0
    ticks = partition.tick_windows(K, win, 5000, 10000)
    t_dev = torch.as_tensor(ticks).cuda()
    zs, cs = [], []
    for m0, m1 in partition.model_blocks(M, n_shards):
        ev = partition.events_for_models(w["events"], m0, m1)
        bprof = tracegen.default_profile(m1 - m0, win)
        sig = partition.block_signal(tre, {"events": _cuda(ev)}, win, K, bprof,
                                     w["slo_ttft_ms"][m0:m1])
        for k in "PDAW":
            np.testing.assert_array_equal(sig["counts"][k].cpu().numpy(), ref[k][:, m0:m1],
                                          err_msg=f"{m0} {k}")
        np.testing.assert_array_equal(sig["theta"].cpu().numpy(), ref["theta"][m0:m1])
        np.testing.assert_array_equal(sig["Z"].cpu().numpy(), ref["Z"][:, m0:m1])
        zs.append(sig["Z"].index_select(0, t_dev))
        cs.append(sig["cls"].index_select(0, t_dev))
    Zt, ct = torch.cat(zs, 1), torch.cat(cs, 1)
    mv, rf, n, _ = partition.walk_on_ticks(tre, Zt, ct, prof, win, 5000, 10000, w["budget"],
                                           w["r0"], w["r_min"], w["footprint"])
    assert n == ref["n_moves"]
    np.testing.assert_array_equal(rf.cpu().numpy(), ref["r_final"])
    np.testing.assert_array_equal(mv, ref["moves"])


def test_sweep_split_by_traces(tre):
    from paper_2609_29160_gb300 import partition
    sw = tracegen.sweep_workload(scale=0.02, n_traces=5, duration_s=600.0)
    alpha = [min(1.0, x / 5000.0) for x in sw["window_ms"]]
    taus, caps = sw["tau_crit"][::2], sw["pacing_cap"][::2]

    def run(traces):
        out = tre.tre_sweep([_cuda(t) for t in traces], sw["M"], sw["duration_ms"],
                            sw["window_ms"], alpha, taus, caps, sw["w_p"], sw["w_q"],
                            sw["tau_surplus"], sw["slo_ttft_ms"], sw["budget"], sw["r0"],
                            sw["r_min"], sw["footprint"], moves_cap=512, want_counts=True)
        n_inst = len(traces) * len(sw["window_ms"]) * len(taus) * len(caps)
        return out, tre.sweep_moves(out, n_inst, 512)

    whole, whole_mv = run(sw["traces"])
    M = sw["M"]
    Ks = [sw["duration_ms"] // int(x) for x in sw["window_ms"]]
    per_trace = sum(Ks) * M
    per_inst = len(sw["window_ms"]) * len(taus) * len(caps)
    for r in range(2):
        mine = partition.sweep_traces(len(sw["traces"]), r, 2)
        part, part_mv = run([sw["traces"][t] for t in mine])
        for j, t in enumerate(mine):
            for k in ("P", "D", "A", "W", "Z", "cls"):
                a = part[k][j * per_trace:(j + 1) * per_trace].cpu().numpy()
                b = whole[k][t * per_trace:(t + 1) * per_trace].cpu().numpy()
                np.testing.assert_array_equal(a, b, err_msg=f"trace {t} {k}")
            np.testing.assert_array_equal(
                part["theta"][j * len(Ks):(j + 1) * len(Ks)].cpu().numpy(),
                whole["theta"][t * len(Ks):(t + 1) * len(Ks)].cpu().numpy())
            for i in range(per_inst):
                np.testing.assert_array_equal(part_mv[j * per_inst + i],
                                              whole_mv[t * per_inst + i])
