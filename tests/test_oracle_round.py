"""Pins of the round oracle (Algorithm 1, Sec. 3.4): frontiers, the budget,
batch collection and candidate rows on hand-built graphs."""
import numpy as np

from helpers import mk
from oracle import oracle as O
from oracle import round as R
from paper_2608_15762_gb300.workloads import random_desc


def test_frontiers_by_hand():
    # 0 -> 1 -> 2, 0 -> 3; 0 done, 1 issued
    d = mk([[], [0], [1], [0]], [1, 1, 1, 1])
    fu, fs = R.frontiers(d, [2, 1, 0, 0])
    assert fu == [2, 3] and fs == [0, 1]
    fu, fs = R.frontiers(d, [0, 0, 0, 0])
    assert fu == [0] and fs == []


def test_budget_and_empty_frontier():
    d = mk([[], [0], [1]], [1, 1, 1])
    info, batch = R.select(d, [1, 0, 0], [0, 0, 0], budget=1, max_batch=8)
    assert info[5] == R.BUDGET and batch == [] and info[3] == 1
    info, batch = R.select(d, [2, 2, 2], [0, 0, 0], budget=4, max_batch=8)
    assert info[5] == R.EMPTY and info[1] == -1 and batch == []


def test_collect_follows_successors_in_id_order():
    # diamond 0 -> {1, 2} -> 3 -> 4, and an unrelated root 5 (more urgent)
    d = mk([[], [0], [0], [1, 2], [3], []], [1] * 6)
    prio = [5, 0, 0, 0, 0, 9]
    info, batch = R.select(d, [0] * 6, prio, budget=100, max_batch=100)
    assert info[1] == 0 and batch == [0, 1, 2, 3, 4]      # 5 is not connected
    info, batch = R.select(d, [0] * 6, prio, budget=100, max_batch=3)
    assert batch == [0, 1, 2] and info[0] == 3
    info, batch = R.select(d, [0] * 6, prio, budget=2, max_batch=100)   # cap = budget - issued
    assert batch == [0, 1]
    # the most urgent frontier op is chosen, ties to the smaller id
    info, _ = R.select(d, [0] * 6, [5, 0, 0, 0, 0, 5], budget=100, max_batch=100)
    assert info[1] == 0


def test_a_successor_waits_for_an_unscheduled_predecessor_outside_the_batch():
    # 0 -> 2 <- 1: 1 is unscheduled and not reachable from 0
    d = mk([[], [], [0, 1]], [1, 1, 1])
    _, batch = R.select(d, [0, 0, 0], [0, 1, 2], budget=10, max_batch=10)
    assert batch == [0]
    _, batch = R.select(d, [0, 2, 0], [0, 1, 2], budget=10, max_batch=10)   # 1 done: 2 follows
    assert batch == [0, 2]


def test_candidate_rows_by_hand():
    place = np.array([3, 3, 3, 3, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0], np.uint8)
    batch = [1, 3]
    part_off, part_dev = [0, 1, 3], [2, 0, 1]          # partitions {2}, {0, 1}
    tmpl, role = [0, 0, 0, 0], [0, 1, 0, 1]
    n_roles = 2
    # template 0: partition 0 maps both roles to slot 0; partition 1 role 0 -> 1, role 1 -> 5 (invalid)
    mapping = [0, 0, 1, 5]
    rows = R.candidate_rows(place, batch, part_off, part_dev, tmpl, role, mapping, n_roles)
    assert rows[0, :4].tolist() == [3, 2, 3, 2]
    assert rows[1, :4].tolist() == [3, 255, 3, 255]


def _closed_states(g, desc, p_sched=0.4):
    pred, _ = R._lists(desc)
    st = np.zeros(desc.n_ops, np.uint8)
    for i in range(desc.n_ops):
        if all(st[q] != 0 for q in pred[i]) and g.random() < p_sched:
            st[i] = 2 if g.random() < 0.6 else 1
    return st


def test_rounds_keep_the_schedule_closed_and_pick_the_best_row():
    g = np.random.default_rng(1)
    d = random_desc(17, 120, 4, dur_hi=60)
    pred, _ = R._lists(d)
    state = _closed_states(g, d)
    place = np.zeros(128, np.uint8)
    place[:120] = g.integers(0, 4, 120)
    prio = g.integers(0, 50, 120)
    tmpl = np.zeros(120, np.int32)
    role = g.integers(0, 3, 120)
    part_off, part_dev = [0, 1, 2, 4, 8], [0, 3, 1, 2, 0, 1, 2, 3]
    mapping = g.integers(0, 2, 4 * 3)
    for _ in range(6):
        info, batch, rows, best, state2, place2 = R.round_step(d, state, place, prio, tmpl, role, part_off,
                                                               part_dev, mapping, 3, budget=40, max_batch=12)
        if info[5] == R.BATCH:
            s, _, _ = O.simulate_batch(d, rows)
            feasible = [k for k in range(rows.shape[0]) if s["status"][k] == 0 and not s["viol_flag"][k]]
            if feasible:
                k = min(feasible, key=lambda k: (int(s["score"][k]), k))
                assert best[0] == k
                assert all(state2[x] == 1 and place2[x] == rows[k, x] for x in batch)
        for i in range(120):
            if state2[i]:
                assert all(state2[q] for q in pred[i])
        state, place = state2, place2
        state[state == 1] = np.where(g.random(int((state == 1).sum())) < 0.5, 2, 1)   # some finish


def test_collection_takes_the_smallest_waiting_id():
    # 0 -> {1, 3}, 1 -> 2: after 0 and 1, op 2 (smaller id) comes before op 3
    d = mk([[], [0], [1], [0]], [1] * 4)
    _, batch = R.select(d, [0] * 4, [0, 1, 2, 3], budget=10, max_batch=3)
    assert batch == [0, 1, 2]
    _, batch = R.select(d, [0] * 4, [0, 1, 2, 3], budget=10, max_batch=10)
    assert batch == [0, 1, 2, 3]
