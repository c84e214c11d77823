"""Independent restatements of the simulation semantics, used to pin the oracle.

Nothing here is imported by the product.  Each formulation is written from the
definitions (Sec. 3.3 of the paper, with the readings listed in the design
notes) without looking at the oracle's event loop:

* ``tick_sim``: advances time one microsecond at a time.  At each tick it
  completes running ops, then marks ops whose every input is present, then
  lets each idle accelerator start its ready op with the smallest
  (ready time, id).  Only usable for small durations.
* ``sweep_sim``: the priority-sweep restatement: ops are taken in global
  (ready time, id) order from a heap of ops whose predecessors are all
  finished, and each starts at max(ready, accelerator free time).
* ``copies`` / ``memory_brute``: HBM copy intervals [alloc, free) derived
  from the residency rules, and live memory evaluated directly at every
  instant where it can change.
* ``tick_sim_arb``: the tick simulation with arbitrated transfers (Sec.
  3.5.2): at each microsecond, completions free their endpoints and links,
  finished producers raise one intent per remote accelerator, and pending
  intents start, in (intent time, producer, destination) order, whenever
  their sending endpoint, receiving endpoint and link are free.
"""
from __future__ import annotations

import heapq
from typing import Dict, List

import numpy as np

INT64_MAX = np.iinfo(np.int64).max


def lists(desc):
    n = desc.n_ops
    pred = [desc.pred_idx[desc.pred_off[i]:desc.pred_off[i + 1]].tolist() for i in range(n)]
    succ = [[] for _ in range(n)]
    for i in range(n):
        for p in pred[i]:
            succ[p].append(i)
    if desc.cons_off is None:
        cons = [list(s) for s in succ]
    else:
        cons = [desc.cons_idx[desc.cons_off[i]:desc.cons_off[i + 1]].tolist() for i in range(n)]
    return pred, succ, cons


def xfer(desc, d, e, b):
    if d == e:
        return 0
    bw = int(desc.bw[d * desc.n_dev + e])
    lat = int(desc.lat[d * desc.n_dev + e])
    return -(-int(b) // bw) + lat


def tick_sim(desc, place, t_max=100000):
    """Returns (ready, start, finish) lists."""
    n, D = desc.n_ops, desc.n_dev
    pred, succ, _ = lists(desc)
    dev = [int(x) for x in place[:n]]
    ready = [None] * n
    start = [None] * n
    finish = [None] * n
    running = [None] * D
    done = 0
    t = 0
    while done < n:
        assert t <= t_max, "tick simulation did not finish"
        for d in range(D):
            i = running[d]
            if i is not None and finish[i] == t:
                running[d] = None
                done += 1
        for i in range(n):
            if ready[i] is not None:
                continue
            ok = t >= int(desc.release[i])
            for p in pred[i]:
                if finish[p] is None or finish[p] > t or \
                        t < finish[p] + xfer(desc, dev[p], dev[i], desc.out_bytes[p]):
                    ok = False
                    break
            if ok:
                ready[i] = t
        for d in range(D):
            if running[d] is not None or t < int(desc.avail0[d]):
                continue
            cands = [(ready[i], i) for i in range(n)
                     if dev[i] == d and ready[i] is not None and start[i] is None]
            if cands:
                _, i = min(cands)
                start[i] = t
                finish[i] = t + desc.dur_on(i, d)
                running[d] = i
        t += 1
    return ready, start, finish


def sweep_sim(desc, place):
    n, D = desc.n_ops, desc.n_dev
    pred, succ, _ = lists(desc)
    dev = [int(x) for x in place[:n]]
    free = [int(x) for x in desc.avail0]
    ready = [None] * n
    start = [None] * n
    finish = [None] * n
    left = [len(p) for p in pred]
    heap = []
    for i in range(n):
        if not pred[i]:
            ready[i] = int(desc.release[i])
            heapq.heappush(heap, (ready[i], i))
    last_key = None
    while heap:
        r, i = heapq.heappop(heap)
        assert last_key is None or (r, i) > last_key
        last_key = (r, i)
        d = dev[i]
        start[i] = max(r, free[d])
        finish[i] = start[i] + desc.dur_on(i, d)
        free[d] = finish[i]
        for j in succ[i]:
            left[j] -= 1
            if left[j] == 0:
                rj = int(desc.release[j])
                for p in pred[j]:
                    rj = max(rj, finish[p] + xfer(desc, dev[p], dev[j], desc.out_bytes[p]))
                ready[j] = rj
                heapq.heappush(heap, (rj, j))
    return ready, start, finish


def link_of(desc, d, e):
    D = desc.n_dev
    return d * D + e if desc.link_id is None else int(desc.link_id[d * D + e])


def tick_sim_arb(desc, place, t_max=100000):
    """Returns (ready, start, finish, transfers); transfers: dicts with p, e,
    intent, start, done."""
    n, D = desc.n_ops, desc.n_dev
    pred, succ, _ = lists(desc)
    dev = [int(x) for x in place[:n]]
    ready = [None] * n
    start = [None] * n
    finish = [None] * n
    running = [None] * D
    xs = {}            # (p, e) -> transfer
    done_ops = 0
    t = 0
    while done_ops < n:
        assert t <= t_max, "tick simulation did not finish"
        for d in range(D):
            i = running[d]
            if i is not None and finish[i] == t:
                running[d] = None
                done_ops += 1
                for e in sorted({dev[j] for j in succ[i] if dev[j] != d}):
                    xs[(i, e)] = dict(p=i, e=e, intent=t, start=None, done=None)
        # arbitration, repeated while a transfer completes at this tick
        while True:
            active = [x for x in xs.values() if x["start"] is not None and x["done"] > t]
            pend = sorted((x for x in xs.values() if x["start"] is None),
                          key=lambda x: (x["intent"], x["p"], x["e"]))
            started = False
            for x in pend:
                src = dev[x["p"]]
                clash = any(dev[y["p"]] == src or y["e"] == x["e"] or
                            link_of(desc, dev[y["p"]], y["e"]) == link_of(desc, src, x["e"])
                            for y in active)
                if not clash:
                    x["start"] = t
                    x["done"] = t + xfer(desc, src, x["e"], desc.out_bytes[x["p"]])
                    active.append(x)
                    started = True
            if not (started and any(x["done"] == t for x in active)):
                break
        for i in range(n):
            if ready[i] is not None:
                continue
            ok = t >= int(desc.release[i])
            for p in pred[i]:
                if finish[p] is None or finish[p] > t:
                    ok = False
                elif dev[p] != dev[i]:
                    x = xs.get((p, dev[i]))
                    ok = ok and x is not None and x["done"] is not None and x["done"] <= t
                if not ok:
                    break
            if ok:
                ready[i] = t
        for d in range(D):
            if running[d] is not None or t < int(desc.avail0[d]):
                continue
            cands = [(ready[i], i) for i in range(n)
                     if dev[i] == d and ready[i] is not None and start[i] is None]
            if cands:
                _, i = min(cands)
                start[i] = t
                finish[i] = t + desc.dur_on(i, d)
                running[d] = i
        t += 1
    xl = sorted(xs.values(), key=lambda x: (x["intent"], x["p"], x["e"]))
    return ready, start, finish, xl


def copies(desc, place, start, finish, transfers=None) -> List[Dict]:
    """Every HBM copy as {dev, op, bytes, alloc, free}.  Without
    ``transfers`` a remote copy is allocated at the producer's finish and
    arrives one transfer estimate later; with them (arbitrated transfers) it
    is allocated when its transfer starts and arrives when it is done."""
    n = desc.n_ops
    pred, succ, cons = lists(desc)
    dev = [int(x) for x in place[:n]]
    tx = {} if transfers is None else {(x["p"], x["e"]): x for x in transfers}
    out = []
    for i in range(n):
        b = int(desc.out_bytes[i])
        d = dev[i]
        remote = sorted({dev[j] for j in succ[i] if dev[j] != d})
        if transfers is None:
            alloc = {e: finish[i] for e in remote}
            arrive = {e: finish[i] + xfer(desc, d, e, b) for e in remote}
        else:
            alloc = {e: tx[(i, e)]["start"] for e in remote}
            arrive = {e: tx[(i, e)]["done"] for e in remote}
        src_free = max([finish[i]] + list(arrive.values()) +
                       [finish[c] for c in cons[i] if dev[c] == d])
        out.append(dict(dev=d, op=i, bytes=b, alloc=start[i], free=src_free))
        for e in remote:
            t_free = max([arrive[e]] + [finish[c] for c in cons[i] if dev[c] == e])
            out.append(dict(dev=e, op=i, bytes=b, alloc=alloc[e], free=t_free))
    return out


def memory_brute(desc, place, start, finish, transfers=None):
    """Peak per device and first violation (time, op, dev) by evaluating live
    memory directly from the copy intervals at every time where it can change
    (every alloc and free instant; it is constant in between).  At an instant
    t the live set is base + copies with alloc < t < free, then the copies
    allocated at t are added in op order; the first one that leaves the total
    above capacity is that device's violation at t."""
    D = desc.n_dev
    cps = copies(desc, place, start, finish, transfers)
    peak = [int(desc.base[d]) for d in range(D)]
    viol = None
    for d in range(D):
        mine = [c for c in cps if c["dev"] == d]
        cap = int(desc.cap[d])
        instants = sorted({c["alloc"] for c in mine} | {c["free"] for c in mine})
        for t in instants:
            live = int(desc.base[d]) + sum(
                c["bytes"] for c in mine if c["alloc"] < t and c["free"] > t)
            assert live >= 0
            allocs = sorted((c["op"], c["bytes"], c["free"]) for c in mine if c["alloc"] == t)
            for op, b, fr in allocs:
                assert fr > t or b == 0
                live += b
                if live > cap and (viol is None or (t, op, d) < viol):
                    viol = (t, op, d)
            peak[d] = max(peak[d], live)
    return peak, viol


def summarize(desc, place, start, finish, ready=None, transfers=None):
    """Summary dict computed from a schedule by the stated definitions."""
    n = desc.n_ops
    peak, viol = memory_brute(desc, place, start, finish, transfers)
    R = desc.n_req
    done = [0] * R
    for i in range(n):
        r = int(desc.req_id[i])
        if r >= 0:
            done[r] = max(done[r], finish[i])
    miss = sum(1 for r in range(R) if done[r] > int(desc.deadline[r]))
    score = sum(finish[i] for i in range(n) if desc.scored[i])
    return dict(status=0, viol_flag=int(viol is not None),
                viol_time=-1 if viol is None else viol[0],
                viol_op=-1 if viol is None else viol[1],
                viol_dev=-1 if viol is None else viol[2],
                makespan=max(finish) if n else 0,
                score=INT64_MAX if viol is not None else score,
                sla_miss=miss, events=n, peak=peak, req_done=done)
