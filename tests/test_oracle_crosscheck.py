"""The oracle's event loop agrees with two independent formulations: a
tick-stepped simulator and the priority-sweep restatement (each accelerator
runs its ops in (ready, id) order, start = max(ready, queue free time)).
Every fourth seed uses 2-3 accelerator types with per-type durations."""
import numpy as np
import pytest

import refsim
from helpers import row, summary_dict
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import random_desc


def _rand(seed, n_hi=24, d_hi=4, dur_hi=12):
    g = np.random.default_rng(10_000 + seed)
    n = int(g.integers(1, n_hi))
    D = int(g.integers(1, d_hi + 1))
    d = random_desc(seed, n, D, dur_hi=dur_hi, bytes_hi=64, explicit_cons=bool(seed % 2),
                    link_hetero=bool(seed % 3), n_types=(2 + seed % 2) if seed % 4 == 3 else 0)
    # small links so transfers matter at these time scales
    d.bw[:] = np.random.default_rng(seed).integers(4, 40, d.bw.shape[0])
    d.lat[:] = np.random.default_rng(seed + 1).integers(0, 6, d.lat.shape[0])
    place = g.integers(0, D, n)
    return d, place


@pytest.mark.parametrize("block", range(8))
def test_tick_stepped_equals_oracle(block):
    for seed in range(block * 40, block * 40 + 40):
        d, place = _rand(seed)
        rd, st, fi = refsim.tick_sim(d, place)
        r = O.simulate(d, row(place))
        assert r["ready"].tolist() == rd, seed
        assert r["start"].tolist() == st, seed
        assert r["finish"].tolist() == fi, seed
        want = refsim.summarize(d, place, st, fi)
        for k in ("viol_flag", "viol_time", "viol_op", "viol_dev", "makespan", "score",
                  "sla_miss", "events"):
            assert r[k] == want[k], (seed, k)
        assert r["peak"].tolist() == want["peak"]
        assert r["req_done"].tolist() == want["req_done"]


@pytest.mark.parametrize("block", range(10))
def test_priority_sweep_equals_oracle(block):
    for seed in range(block * 300, block * 300 + 300):
        d, place = _rand(seed, n_hi=120, d_hi=8, dur_hi=2000)
        rd, st, fi = refsim.sweep_sim(d, place)
        r = O.simulate(d, row(place))
        assert r["start"].tolist() == st, seed
        assert r["finish"].tolist() == fi, seed
        assert r["ready"].tolist() == rd, seed


def test_batch_equals_single_candidate_calls():
    d = random_desc(5, 70, 4)
    g = np.random.default_rng(5)
    place = np.zeros((33, 80), np.uint8)
    place[:, :70] = g.integers(0, 4, (33, 70))
    place[7, 3] = 9   # an invalid device id in one row
    s, peak, req = O.simulate_batch(d, place, nthreads=3)
    for k in range(33):
        r = O.simulate(d, place[k])
        assert summary_dict(s[k]) == {kk: r[kk] for kk in summary_dict(s[k])}
        assert peak[k].tolist() == r["peak"].tolist()
        assert req[k].tolist() == r["req_done"].tolist()
    assert s[7]["status"] == O.SIM_BADDEV
