"""Incremental what-if (Sec. 3.4.2): a candidate given as moves against a
base placement equals the full simulation of the moved placement; the
operators whose base ready time is below the resume time T0 keep their base
schedule exactly, and so does every HBM event before T0."""
import numpy as np
import pytest

import refsim
from helpers import summary_dict
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import Moves, random_desc, random_moves


def _applied(base, moves, k):
    p = base.copy()
    for m in range(moves.off[k], moves.off[k + 1]):
        p[moves.op[m]] = moves.dev[m]
    return p


def _t0(d, base, moves, k, base_finish):
    pred, _, _ = refsim.lists(d)
    t0 = None
    for m in range(moves.off[k], moves.off[k + 1]):
        x = int(moves.op[m])
        if int(moves.dev[m]) == int(base[x]):
            continue
        t = min(base_finish[p] for p in pred[x]) if pred[x] else int(d.release[x])
        t0 = t if t0 is None else min(t0, t)
    return t0


@pytest.mark.parametrize("seed", range(16))
def test_incremental_equals_full_simulation_of_applied_moves(seed):
    g = np.random.default_rng(seed)
    n = int(g.integers(1, 120))
    D = int(g.integers(1, 7))
    d = random_desc(3000 + seed, n, D, explicit_cons=bool(seed % 2), dur_hi=200)
    base = g.integers(0, D, n).astype(np.uint8)
    mv = random_moves(seed, 40, base, D, max_moves=6)
    s, peak, req = O.incremental_batch(d, base, mv, nthreads=2)
    rows = np.zeros((40, max(16, (n + 15) // 16 * 16)), np.uint8)
    for k in range(40):
        rows[k, :n] = _applied(base, mv, k)
    s2, peak2, req2 = O.simulate_batch(d, rows, nthreads=2)
    # independent base schedule from the priority-sweep restatement
    b_ready, b_start, b_finish = refsim.sweep_sim(d, base)
    for k in range(40):
        a, b = summary_dict(s[k]), summary_dict(s2[k])
        ev = a.pop("events")
        b.pop("events")
        assert a == b
        assert peak[k].tolist() == peak2[k].tolist()
        assert req[k].tolist() == req2[k].tolist()
        t0 = _t0(d, base, mv, k, b_finish)
        want = 0 if t0 is None else sum(1 for i in range(n) if b_ready[i] >= t0)
        assert ev == want


@pytest.mark.parametrize("seed", range(16))
def test_prefix_before_t0_is_unchanged(seed):
    """The property the incremental kernels rely on: ops with base ready time
    < T0 keep (ready, start, finish), and HBM events at times < T0 are the
    same, so a base snapshot taken before T0 is a valid resume point."""
    g = np.random.default_rng(500 + seed)
    n = int(g.integers(5, 150))
    D = int(g.integers(2, 7))
    d = random_desc(4000 + seed, n, D, explicit_cons=bool(seed % 2), dur_hi=300)
    base = g.integers(0, D, n).astype(np.uint8)
    mv = random_moves(100 + seed, 30, base, D, max_moves=5, allow_noop=False)
    rb = O.simulate(d, base)
    for k in range(30):
        t0 = _t0(d, base, mv, k, rb["finish"].tolist())
        if t0 is None:
            continue
        p = _applied(base, mv, k)
        rc = O.simulate(d, p)
        for i in range(n):
            if rb["ready"][i] < t0:
                assert rc["ready"][i] == rb["ready"][i]
                assert rc["start"][i] == rb["start"][i]
                assert rc["finish"][i] == rb["finish"][i]
            else:
                assert rc["ready"][i] >= t0
        ev_b = sorted((c["dev"], c["op"], c["alloc"], c["free"], c["bytes"]) for c in refsim.copies(
            d, base, rb["start"].tolist(), rb["finish"].tolist()))
        ev_c = sorted((c["dev"], c["op"], c["alloc"], c["free"], c["bytes"]) for c in refsim.copies(
            d, p, rc["start"].tolist(), rc["finish"].tolist()))

        def before(evs):
            out = set()
            for (dv, op, a, f, by) in evs:
                if a < t0:
                    out.add((dv, op, "a", a, by))
                if f < t0:
                    out.add((dv, op, "f", f, by))
            return out
        assert before(ev_b) == before(ev_c)


def test_move_status_codes():
    d = random_desc(1, 10, 3)
    base = np.zeros(10, np.uint8)
    mv = Moves(np.array([0, 0, 2, 4, 5, 6], np.int32),
               np.array([1, 2, 3, 3, 11, 4], np.int32),
               np.array([1, 2, 1, 2, 0, 3], np.uint8))
    s, _, _ = O.incremental_batch(d, base, mv, nthreads=1)
    assert s["status"].tolist() == [0, 0, O.SIM_MOVE_DUP, O.SIM_MOVE_RANGE, O.SIM_MOVE_RANGE]
    full = O.simulate(d, base)
    assert s[0]["events"] == 0 and s[0]["score"] == full["score"]
    bad = base.copy()
    bad[4] = 7
    s, _, _ = O.incremental_batch(d, bad, mv, nthreads=1)
    assert (s["status"] == O.SIM_BADBASE).all()
