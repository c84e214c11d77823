"""Pins of the oracle's heterogeneous accelerators: the operator estimator is
kept per (accelerator type, operator) (Sec. 3.3.1), so an op's duration is the
one of the type of the accelerator it is placed on."""
import dataclasses

import numpy as np
import pytest

from helpers import mk, row
from oracle import oracle as O
from paper_2608_15762_gb300.workloads import random_desc


def typed(desc, dev_type, dur_by_type):
    return dataclasses.replace(desc, dev_type=np.asarray(dev_type, np.uint8),
                               dur_by_type=np.asarray(dur_by_type, np.int64)).normalized()


def test_hand_computed_chain_across_two_types():
    # op0 -> op1 -> op2; accelerator 0 has type 0, accelerator 1 type 1;
    # transfers: ceil(bytes / 100) + 3
    d = mk([[], [0], [1]], [1, 1, 1], [200, 100, 0], n_dev=2, bw=100, lat=3)
    d = typed(d, [0, 1], [[10, 25], [30, 12], [5, 9]])
    # [0, 1, 1]: op0 0..10 on type 0; arrives at 10 + 2 + 3 = 15; op1 15..27 on
    # type 1; op2 local, 27..36
    r = O.simulate(d, row([0, 1, 1]))
    assert r["start"].tolist() == [0, 15, 27] and r["finish"].tolist() == [10, 27, 36]
    # [1, 0, 0]: op0 0..25 on type 1; arrives at 30; op1 30..60; op2 60..65
    r = O.simulate(d, row([1, 0, 0]))
    assert r["start"].tolist() == [0, 30, 60] and r["finish"].tolist() == [25, 60, 65]
    assert r["score"] == 25 + 60 + 65


@pytest.mark.parametrize("seed", range(10))
def test_chain_on_one_accelerator_sums_its_type_durations(seed):
    g = np.random.default_rng(seed)
    n, T = int(g.integers(1, 30)), int(g.integers(2, 5))
    D = int(g.integers(1, 6))
    d = mk([[i - 1] if i else [] for i in range(n)], [1] * n, g.integers(0, 1000, n), n_dev=D,
           bw=7, lat=2)
    types = g.integers(0, T, D)
    table = g.integers(1, 500, (n, T))
    d = typed(d, types, table)
    for dev in range(D):
        r = O.simulate(d, row([dev] * n))
        durs = table[:, types[dev]]
        assert r["makespan"] == int(durs.sum())
        assert r["finish"].tolist() == np.cumsum(durs).tolist()


@pytest.mark.parametrize("seed", range(8))
def test_equal_columns_reduce_to_one_type(seed):
    d = random_desc(300 + seed, 60, 5, dur_hi=400, explicit_cons=bool(seed % 2))
    T = 3
    h = typed(d, np.random.default_rng(seed).integers(0, T, 5), np.repeat(d.dur[:, None], T, axis=1))
    place = np.zeros((16, 64), np.uint8)
    place[:, :60] = np.random.default_rng(seed).integers(0, 5, (16, 60))
    a = O.simulate_batch(d, place)
    b = O.simulate_batch(h, place)
    for x, y in zip(a, b):
        assert np.array_equal(x, y)


def test_a_type_only_matters_where_it_is_used():
    # the slow type's durations change nothing for a placement that never uses it
    d = random_desc(77, 50, 4, dur_hi=300)
    types = [0, 0, 1, 1]
    table = np.stack([d.dur, d.dur * 7], axis=1)
    h = typed(d, types, table)
    place = np.zeros(64, np.uint8)
    place[:50] = np.random.default_rng(1).integers(0, 2, 50)   # accelerators 0, 1 only
    assert O.simulate(d, place)["finish"].tolist() == O.simulate(h, place)["finish"].tolist()
    place[:50] = np.random.default_rng(1).integers(2, 4, 50)   # the slow pair only
    slow = O.simulate(h, place)
    fast = O.simulate(typed(d, types, np.stack([d.dur, d.dur], axis=1)), place)
    assert slow["makespan"] > fast["makespan"]


def test_type_validation():
    d = mk([[], [0]], [3, 4], n_dev=2)
    assert O.check(typed(d, [0, 1], [[1, 2], [3, 4]])) == 0
    assert O.check(typed(d, [0, 2], [[1, 2], [3, 4]])) == O.EINVAL   # type id >= T
    assert O.check(typed(d, [0, 1], [[1, 0], [3, 4]])) == O.EINVAL   # duration < 1
    one = typed(d, [0, 0], [[9], [9]])                               # one type: dur_us applies
    assert O.simulate(one, row([0, 0]))["finish"].tolist() == [3, 7]
