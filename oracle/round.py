"""CPU oracle of one scheduling round (Algorithm 1, Sec. 3.4).

TEST INFRASTRUCTURE ONLY: the plain restatement the GPU round kernels are
checked against; the product never imports it.

Steps, in Algorithm 1's order:

* Frontiers (Sec. 3.4.1): op states 0 unscheduled, 1 issued, 2 done.  The
  scheduled frontier holds issued/done ops with an unscheduled successor; the
  unscheduled frontier F_u holds unscheduled ops whose predecessors are all
  issued or done.
* If the issued count is at least the budget B, or F_u is empty, the round
  schedules nothing.
* op = the highest-priority op of F_u: smallest (priority, op id).
* Batch = CollectConnectedGraph(op, B): candidates are taken in increasing op
  id starting from {op}; taking x adds each unscheduled successor of x all of
  whose predecessors are scheduled, taken or waiting; at most
  min(max_batch, B - issued) ops are taken.
* CandidatePartitions: for each pre-defined partition p (an ordered list of
  accelerators) the batch op x goes to accelerator
  part_dev[p][map[tmpl[x]][p][role[x]]] (255 if that slot is outside the
  partition); every other op keeps its current placement.
* Each candidate is simulated (the simulation oracle, in parallel in the
  paper's wording); the best feasible one by select_best wins; its placement
  is written back and the batch becomes issued.
"""
from __future__ import annotations

import heapq

import numpy as np

from oracle import oracle as O

BATCH, BUDGET, EMPTY, NO_FEASIBLE = 0, 1, 2, 3


def _lists(desc):
    n = desc.n_ops
    pred = [desc.pred_idx[desc.pred_off[i]:desc.pred_off[i + 1]].tolist() for i in range(n)]
    succ = [[] for _ in range(n)]
    for i in range(n):
        for p in pred[i]:
            succ[p].append(i)
    return pred, succ


def frontiers(desc, state):
    pred, succ = _lists(desc)
    fu = [i for i in range(desc.n_ops) if state[i] == 0 and all(state[p] != 0 for p in pred[i])]
    fs = [i for i in range(desc.n_ops) if state[i] != 0 and any(state[j] == 0 for j in succ[i])]
    return fu, fs


def select(desc, state, prio, budget, max_batch):
    """Returns (info list of 8, batch list)."""
    fu, fs = frontiers(desc, state)
    issued = int(np.sum(np.asarray(state) == 1))
    chosen = min(fu, key=lambda i: (int(prio[i]), i)) if fu else -1
    info = [0, chosen, len(fu), issued, len(fs), BATCH, 0, 0]
    if issued >= budget:
        info[5] = BUDGET
        return info, []
    if not fu:
        info[5] = EMPTY
        return info, []
    pred, succ = _lists(desc)
    cap = min(max_batch, budget - issued)
    marked = {chosen}
    heap = [chosen]
    batch = []
    while heap and len(batch) < cap:
        x = heapq.heappop(heap)
        batch.append(x)
        for j in succ[x]:
            if state[j] == 0 and j not in marked and all(state[p] != 0 or p in marked for p in pred[j]):
                marked.add(j)
                heapq.heappush(heap, j)
    info[0] = len(batch)
    return info, batch


def candidate_rows(place, batch, part_off, part_dev, tmpl, role, mapping, n_roles):
    n_part = len(part_off) - 1
    rows = np.tile(np.asarray(place, np.uint8), (n_part, 1))
    for p in range(n_part):
        size = part_off[p + 1] - part_off[p]
        for x in batch:
            s = int(mapping[(int(tmpl[x]) * n_part + p) * n_roles + int(role[x])])
            rows[p, x] = part_dev[part_off[p] + s] if 0 <= s < size else 255
    return rows


def round_step(desc, state, place, prio, tmpl, role, part_off, part_dev, mapping, n_roles, budget, max_batch,
               score_mode=0):
    """One round; returns (info, batch, rows, best, new_state, new_place)."""
    state = np.array(state, np.uint8)
    place = np.array(place, np.uint8)
    info, batch = select(desc, state, prio, budget, max_batch)
    rows = candidate_rows(place, batch, part_off, part_dev, tmpl, role, mapping, n_roles)
    best = None
    if info[5] == BATCH:
        s, _, _ = O.simulate_batch(desc, rows)
        best = O.select_best(s, score_mode)
        if best[0] < 0:
            info[5] = NO_FEASIBLE
        else:
            for x in batch:
                place[x] = rows[best[0], x]
                state[x] = 1
    return info, batch, rows, best, state, place
