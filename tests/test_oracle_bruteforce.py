"""Brute force over every placement of DAGs with at most 8 ops on 2
accelerators (Algorithm 1: discard OOM placements, keep the smallest average
completion time, ties to the lowest candidate index)."""
import itertools

import numpy as np
import pytest

import refsim
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import INT64_MAX, random_desc


def _all_rows(n):
    rows = np.zeros((2 ** n, 16), np.uint8)
    for k, bits in enumerate(itertools.product((0, 1), repeat=n)):
        rows[k, :n] = bits
    return rows


@pytest.mark.parametrize("seed", range(24))
def test_select_best_is_the_exhaustive_argmin(seed):
    g = np.random.default_rng(seed)
    n = int(g.integers(1, 9))
    d = random_desc(900 + seed, n, 2, dur_hi=9, bytes_hi=32, explicit_cons=bool(seed % 2))
    d.bw[:] = g.integers(2, 12, 4)
    d.lat[:] = g.integers(0, 4, 4)
    # tight capacities so that some placements are infeasible
    d.cap[:] = g.integers(24, 90, 2)
    d.base[:] = np.minimum(d.base, d.cap)
    rows = _all_rows(n)
    s, peak, req = O.simulate_batch(d, rows, nthreads=2)
    want_scores, want_miss = [], []
    for k in range(rows.shape[0]):
        _, st, fi = refsim.tick_sim(d, rows[k])
        w = refsim.summarize(d, rows[k], st, fi)
        assert s[k]["score"] == w["score"] and s[k]["viol_flag"] == w["viol_flag"]
        assert peak[k].tolist() == w["peak"]
        want_scores.append(w["score"] if not w["viol_flag"] else None)
        want_miss.append(w["sla_miss"])
    feas = [k for k in range(len(want_scores)) if want_scores[k] is not None]
    want0 = min(feas, key=lambda k: (want_scores[k], k)) if feas else -1
    want1 = min(feas, key=lambda k: (want_miss[k], want_scores[k], k)) if feas else -1
    k0, b0 = O.select_best(s, 0)
    k1, b1 = O.select_best(s, 1)
    assert k0 == want0 and k1 == want1
    assert b0 == (want_scores[want0] if feas else INT64_MAX)


@pytest.mark.parametrize("seed", range(12))
def test_swapping_two_identical_accelerators_is_a_relabeling(seed):
    g = np.random.default_rng(50 + seed)
    n = int(g.integers(1, 9))
    d = random_desc(700 + seed, n, 2, dur_hi=20, bytes_hi=64, with_avail0=False)
    d.bw[:] = int(g.integers(2, 9))
    d.lat[:] = int(g.integers(0, 5))
    d.cap[:] = int(g.integers(40, 200))
    d.base[:] = int(g.integers(0, 20))
    rows = _all_rows(n)
    s, peak, req = O.simulate_batch(d, rows, nthreads=2)
    m = rows.shape[0] - 1
    for k in range(rows.shape[0]):
        c = m - k   # complemented placement: every op on the other accelerator
        for f in ("makespan", "score", "sla_miss", "viol_flag", "viol_op", "viol_time"):
            assert s[k][f] == s[c][f]
        assert peak[k].tolist() == peak[c][::-1].tolist()
        if s[k]["viol_flag"]:
            assert s[k]["viol_dev"] == 1 - s[c]["viol_dev"]
