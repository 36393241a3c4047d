"""Input realism of the workload generator (not parity): a flat-rate model is
an M/M/c queue, so its share of requests that wait and its mean wait follow the
Erlang C formula; the integer-millisecond latent queue agrees with the
generator's records; the per-model FCFS queue never runs more requests than it
has servers."""
import math

import numpy as np
import pytest

import tracegen


def _erlang_c(c, a):
    """Probability that an arrival waits in M/M/c with offered load a < c."""
    s = sum(a ** k / math.factorial(k) for k in range(c))
    top = a ** c / math.factorial(c) * c / (c - a)
    return top / (s + top)


def _flat_spec(c, rho, n_target, seed):
    return tracegen.TraceSpec(n_models=1, duration_s=20000.0, n_target=n_target,
                              cost=np.array([1.0]), share=np.array([1.0]),
                              len_in=np.array([(6.0, 1.0)]), len_out=np.array([(5.0, 0.8)]),
                              budget=c, r0=np.array([c]), rho=rho, rho_mode="max", seed=seed)


@pytest.mark.parametrize("c,rho", [(1, 0.6), (4, 0.8), (8, 0.85)])
def test_flat_rate_queue_follows_erlang_c(c, rho):
    req = tracegen.gen_requests(_flat_spec(c, rho, 40000, seed=11 + c))
    wait = (req["t_start_ms"] - req["t_arr_ms"]).astype(np.float64)
    svc = (req["t_end_ms"] - req["t_start_ms"]).astype(np.float64)
    a = rho * c                                   # offered load in servers
    pc = _erlang_c(c, a)
    # drop the first tenth (the queue starts empty)
    cut = len(wait) // 10
    assert abs((wait[cut:] > 0).mean() - pc) < 0.04
    mean_wait = pc * svc.mean() / (c - a)
    assert abs(wait[cut:].mean() - mean_wait) < 0.15 * mean_wait


def test_latent_queue_agrees_with_the_records():
    spec = tracegen.spec_mid(scale=0.01, seed=3, duration_s=600.0)
    req = tracegen.gen_requests(spec)
    lat = tracegen.gen_latent(spec)
    fc = tracegen.fcfs_records(lat, spec.n_models, lat["r0"])
    assert np.array_equal(lat["model"], req["model"])
    assert np.array_equal(lat["t_arr_ms"], req["t_arr_ms"])
    # whole-millisecond service in place of exact floats: the rounding (half a
    # millisecond per request at most) accumulates only over a busy period
    d = np.abs(fc["t_start_ms"].astype(np.int64) - req["t_start_ms"])
    assert np.median(d) <= 1 and np.percentile(d, 99) <= 12 and d.max() <= 50


def test_fcfs_never_exceeds_its_servers():
    spec = tracegen.spec_mid(scale=0.01, seed=4, duration_s=600.0)
    lat = tracegen.gen_latent(spec)
    fc = tracegen.fcfs_records(lat, spec.n_models, lat["r0"])
    for m in range(spec.n_models):
        sel = fc["model"] == m
        s, e = fc["t_start_ms"][sel].astype(np.int64), fc["t_end_ms"][sel].astype(np.int64)
        a = fc["t_arr_ms"][sel]
        assert (s >= a).all()
        assert (np.diff(s) >= 0).all()            # first come, first served
        ev = np.concatenate([np.stack([s, np.ones_like(s)], 1), np.stack([e, -np.ones_like(e)], 1)])
        ev = ev[np.lexsort((ev[:, 1], ev[:, 0]))]   # ends before starts at equal times
        assert np.cumsum(ev[:, 1]).max() <= int(lat["r0"][m])
