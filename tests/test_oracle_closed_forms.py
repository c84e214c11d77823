"""Closed forms that pin the CPU oracle (Sec. 3.3 semantics)."""
import numpy as np
import pytest

from helpers import mk, row
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import INT64_MAX


def ceil_div(a, b):
    return -(-a // b)


@pytest.mark.parametrize("seed", range(20))
def test_chain_on_one_device_makespan_is_sum_of_durations(seed):
    g = np.random.default_rng(seed)
    n = int(g.integers(1, 40))
    D = int(g.integers(1, 5))
    dur = g.integers(1, 1000, n)
    d = mk([[i - 1] if i else [] for i in range(n)], dur, g.integers(0, 1 << 20, n),
           n_dev=D, bw=g.integers(1, 100), lat=7)
    dev = int(g.integers(0, D))
    r = O.simulate(d, row([dev] * n))
    assert r["makespan"] == int(dur.sum())
    assert r["score"] == int(np.cumsum(dur).sum())
    assert r["start"].tolist() == [0] + np.cumsum(dur)[:-1].tolist()


@pytest.mark.parametrize("seed", range(20))
def test_independent_ops_makespan_is_max_device_load(seed):
    g = np.random.default_rng(100 + seed)
    n = int(g.integers(1, 60))
    D = int(g.integers(1, 6))
    dur = g.integers(1, 500, n)
    d = mk([[] for _ in range(n)], dur, n_dev=D)
    place = g.integers(0, D, n)
    r = O.simulate(d, row(place))
    loads = [int(dur[place == k].sum()) for k in range(D)]
    assert r["makespan"] == max(loads)


@pytest.mark.parametrize("seed", range(20))
def test_alternating_chain_adds_every_crossing_transfer(seed):
    g = np.random.default_rng(200 + seed)
    n = int(g.integers(2, 30))
    dur = g.integers(1, 300, n)
    b = g.integers(0, 1 << 16, n)
    bw, lat = int(g.integers(1, 50)), int(g.integers(0, 20))
    d = mk([[i - 1] if i else [] for i in range(n)], dur, b, n_dev=2, bw=bw, lat=lat)
    place = g.integers(0, 2, n)
    r = O.simulate(d, row(place))
    cross = sum(ceil_div(int(b[i]), bw) + lat for i in range(n - 1) if place[i] != place[i + 1])
    assert r["makespan"] == int(dur.sum()) + cross


@pytest.mark.parametrize("seed", range(20))
def test_fork_join_closed_form(seed):
    g = np.random.default_rng(300 + seed)
    nb = int(g.integers(1, 6))
    D = nb + 1
    # op 0 = source, ops 1..nb = branches, op nb+1 = sink.
    preds = [[]] + [[0] for _ in range(nb)] + [list(range(1, nb + 1))]
    dur = g.integers(1, 400, nb + 2)
    b = g.integers(0, 1 << 16, nb + 2)
    bwm = g.integers(1, 60, (D, D))
    latm = g.integers(0, 30, (D, D))
    d = mk(preds, dur, b, n_dev=D, bw=bwm, lat=latm)
    src_dev = int(g.integers(0, D))
    branch_devs = g.permutation(D)[:nb]           # distinct devices, one may equal src_dev
    place = [src_dev] + branch_devs.tolist() + [src_dev]

    def x(a, c, by):
        return 0 if a == c else ceil_div(int(by), int(bwm[a, c])) + int(latm[a, c])

    expect = int(dur[0]) + max(
        x(src_dev, int(branch_devs[k]), b[0]) + int(dur[1 + k]) + x(int(branch_devs[k]), src_dev, b[1 + k])
        for k in range(nb)) + int(dur[nb + 1])
    r = O.simulate(d, row(place))
    assert r["makespan"] == expect


@pytest.mark.parametrize("seed", range(20))
def test_memory_of_a_one_device_chain(seed):
    g = np.random.default_rng(400 + seed)
    n = int(g.integers(1, 30))
    dur = g.integers(1, 100, n)
    b = g.integers(0, 1 << 30, n)
    base = int(g.integers(0, 1 << 20))
    d = mk([[i - 1] if i else [] for i in range(n)], dur, b, n_dev=3,
           base=[base, 0, 0])
    r = O.simulate(d, row([0] * n))
    expect = max([int(b[0])] + [int(b[i - 1] + b[i]) for i in range(1, n)]) + base
    assert r["peak"][0] == expect
    assert r["peak"][1] == 0 and r["peak"][2] == 0
    assert r["viol_flag"] == 0


def test_capacity_violation_discards_the_placement():
    d = mk([[], [0], [1]], [5, 5, 5], [10, 20, 30], n_dev=1, cap=[49])
    r = O.simulate(d, row([0, 0, 0]))
    # live: [0,10) 10 -> at 5: 10+20 -> at 10: free 10, +30 = 50 > 49.
    assert r["viol_flag"] == 1 and (r["viol_time"], r["viol_op"], r["viol_dev"]) == (10, 2, 0)
    assert r["score"] == INT64_MAX
    assert r["peak"][0] == 50
    d2 = mk([[], [0], [1]], [5, 5, 5], [10, 20, 30], n_dev=1, cap=[50])
    r2 = O.simulate(d2, row([0, 0, 0]))
    assert r2["viol_flag"] == 0 and r2["score"] == 5 + 10 + 15


def test_device_busy_until_avail0_and_release():
    d = mk([[], [0]], [4, 6], n_dev=2, avail0=[10, 0], release=[3, 0])
    r = O.simulate(d, row([0, 0]))
    assert r["start"].tolist() == [10, 14] and r["makespan"] == 20
    r = O.simulate(d, row([1, 1]))
    assert r["start"].tolist() == [3, 7]


def test_queue_starts_earliest_ready_then_lowest_id():
    # ops 0,1,2 independent on one device; 0 and 2 ready at 0, 1 released at 1.
    d = mk([[], [], []], [5, 3, 2], n_dev=1, release=[0, 1, 0])
    r = O.simulate(d, row([0, 0, 0]))
    # t=0: ready {0 (r0), 2 (r0)} -> op 0; t=5: ready {1 (r1), 2 (r0)} -> op 2; then op 1.
    assert r["start"].tolist() == [0, 7, 5]


def test_sla_miss_counts_requests_past_their_deadline():
    d = mk([[], [0], [], [2]], [5, 5, 5, 5], n_dev=2, req_id=[0, 0, 1, 1],
           deadline=[10, 9])
    r = O.simulate(d, row([0, 0, 1, 1]))
    assert r["req_done"].tolist() == [10, 10]
    assert r["sla_miss"] == 1
    r = O.simulate(d, row([0, 0, 0, 0]))
    # op 2 waits for 0; order by (ready, id): 0 (0), 2 (0), 1 (5), 3 (10)
    assert r["start"].tolist() == [0, 10, 5, 15]
    assert r["req_done"].tolist() == [15, 20]
    assert r["sla_miss"] == 2


def test_unscored_ops_do_not_count():
    d = mk([[], [0]], [3, 4], n_dev=1, scored=[0, 1])
    assert O.simulate(d, row([0, 0]))["score"] == 7


def test_bad_device_id_status():
    d = mk([[], [0]], [3, 4], n_dev=2)
    r = O.simulate(d, row([0, 2]))
    assert r["status"] == O.SIM_BADDEV and r["score"] == INT64_MAX and r["events"] == 0


def test_empty_graph():
    d = mk([], [], n_dev=3)
    r = O.simulate(d, row([]))
    assert r["status"] == 0 and r["makespan"] == 0 and r["score"] == 0 and r["events"] == 0
    assert r["peak"].tolist() == [0, 0, 0]
