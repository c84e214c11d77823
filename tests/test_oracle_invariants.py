"""Invariants of the oracle's schedules on random DAGs (Sec. 3.3 semantics)."""
import numpy as np
import pytest

import refsim
from helpers import row
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import random_desc

CASES = [(s, n, D) for s, (n, D) in enumerate(
    [(5, 1), (12, 2), (20, 3), (40, 4), (60, 2), (80, 5), (30, 8), (100, 3)] * 8)]


@pytest.mark.parametrize("seed,n,D", CASES)
def test_schedule_invariants(seed, n, D):
    d = random_desc(seed, n, D, explicit_cons=bool(seed % 2), link_hetero=bool(seed % 3))
    g = np.random.default_rng(seed)
    place = g.integers(0, D, n)
    r = O.simulate(d, row(place))
    assert r["status"] == 0 and r["events"] == n
    pred, succ, cons = refsim.lists(d)
    s, f, rd = r["start"], r["finish"], r["ready"]
    assert (f - s == d.dur).all()
    for i in range(n):
        # ready time = max(release, predecessor arrivals); start not before it
        arr = [int(f[p]) + refsim.xfer(d, place[p], place[i], d.out_bytes[p]) for p in pred[i]]
        assert rd[i] == max([int(d.release[i])] + arr)
        assert s[i] >= rd[i] and s[i] >= d.avail0[place[i]]
    for k in range(D):
        ops = [i for i in range(n) if place[i] == k]
        # queue order is (ready, id); starts follow it, no overlap, and each
        # start is max(ready, previous finish on the queue)
        ops.sort(key=lambda i: (int(rd[i]), i))
        prev = int(d.avail0[k])
        for i in ops:
            assert s[i] == max(int(rd[i]), prev)
            prev = int(f[i])
        load = int(d.dur[place == k].sum())
        if ops:
            assert r["makespan"] >= int(d.avail0[k]) + load
    # makespan bounded below by the contention-free critical path
    est = [0] * n
    for i in range(n):
        est[i] = max([int(d.release[i])] + [est[p] + int(d.dur[p]) for p in pred[i]])
    if n:
        assert r["makespan"] >= max(est[i] + int(d.dur[i]) for i in range(n))
    # memory: every copy's interval is well formed and the peak / first
    # violation equal a direct evaluation of the intervals
    cps = refsim.copies(d, place, s.tolist(), f.tolist())
    for c in cps:
        assert c["free"] >= c["alloc"]
        assert c["free"] > c["alloc"] or c["bytes"] == 0
    peak, viol = refsim.memory_brute(d, place, s.tolist(), f.tolist())
    assert r["peak"].tolist() == peak
    if viol is None:
        assert r["viol_flag"] == 0 and r["viol_op"] == -1
    else:
        assert (r["viol_time"], r["viol_op"], r["viol_dev"]) == viol
