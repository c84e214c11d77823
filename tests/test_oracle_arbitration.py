"""Pins of the oracle's arbitrated-transfer mode (Sec. 3.5.2, "Tensor
Transfer Arbitration"): hand-worked schedules for each kind of conflict
(shared sender, shared receiver, shared link), the arbitration order, the
absence of head-of-line blocking, zero-length transfers, the receive buffer
allocated when its transfer starts; the cases where no two transfers ever
compete (identical to the pure-latency model); agreement with an
independently written tick simulation; and the conflict-freedom, greedy and
FIFO properties of every transfer table on larger random graphs."""
import numpy as np
import pytest

import refsim
from helpers import mk, row
from oracle import oracle as O
from paper_2608_15762_gb300 import workloads as W
from paper_2608_15762_gb300.workloads import random_desc


def _arb(d, place):
    return O.simulate(d, row(place), arbitrated=True)


def _xt(r):
    return [tuple(int(v) for v in x) for x in r["transfers"]]


def test_shared_sender_serializes():
    # op 0 on accelerator 0 feeds op 1 on 1 and op 2 on 2: both transfers
    # leave accelerator 0, so the second waits for the first (10 us each)
    d = mk([[], [0], [0]], [4, 1, 1], out_bytes=[10, 0, 0], n_dev=3, bw=1, lat=0)
    r = _arb(d, [0, 1, 2])
    assert _xt(r) == [(0, 1, 4, 4, 14), (0, 2, 4, 14, 24)]
    assert r["finish"].tolist() == [4, 15, 25]
    assert O.simulate(d, row([0, 1, 2]))["finish"].tolist() == [4, 15, 15]


def test_shared_receiver_serializes_in_producer_order():
    # ops 0 (5 B) and 1 (7 B) finish at 3 on accelerators 0 and 1; op 2 on
    # accelerator 2 needs both: equal intent times go by producer id
    d = mk([[], [], [0, 1]], [3, 3, 2], out_bytes=[5, 7, 0], n_dev=3, bw=1, lat=0)
    r = _arb(d, [0, 1, 2])
    assert _xt(r) == [(0, 2, 3, 3, 8), (1, 2, 3, 8, 15)]
    assert r["ready"][2] == 15 and r["finish"][2] == 17
    # swap the sizes: still producer 0 first (not shortest first)
    d2 = mk([[], [], [0, 1]], [3, 3, 2], out_bytes=[7, 5, 0], n_dev=3, bw=1, lat=0)
    assert _xt(_arb(d2, [0, 1, 2])) == [(0, 2, 3, 3, 10), (1, 2, 3, 10, 15)]


def test_shared_link_serializes_opposite_directions():
    # 0 -> 1 and 1 -> 0 at once: no endpoint is shared, so they overlap,
    # unless both directions are given the same link id
    d = mk([[], [], [0], [1]], [2, 2, 1, 1], out_bytes=[6, 6, 0, 0], n_dev=2, bw=1, lat=0)
    place = [0, 1, 1, 0]
    assert _xt(_arb(d, place)) == [(0, 1, 2, 2, 8), (1, 0, 2, 2, 8)]
    d.link_id = np.array([0, 1, 1, 0], np.int32)
    r = _arb(d, place)
    assert _xt(r) == [(0, 1, 2, 2, 8), (1, 0, 2, 8, 14)]
    assert r["finish"].tolist() == [2, 2, 9, 15]


def test_a_blocked_intent_does_not_block_later_ones():
    # 0 -> 1 (100 us) holds accelerator 1's receiver; 2 -> 1 waits for it, but
    # the later 2 -> 3 starts at once: accelerator 2's sender is not held
    # by a transfer that has not started
    d = mk([[], [], [], [0], [1], [2]], [1, 1, 1, 1, 1, 1], out_bytes=[100, 5, 5, 0, 0, 0],
           n_dev=4, bw=1, lat=0)
    place = [0, 2, 2, 1, 1, 3]
    r = _arb(d, place)
    assert _xt(r) == [(0, 1, 1, 1, 101), (1, 1, 1, 101, 106), (2, 3, 2, 2, 7)]
    assert r["finish"].tolist() == [1, 1, 2, 102, 107, 8]


def test_latency_counts_towards_the_hold():
    # per-pair latency is part of the transfer time, and the sender stays
    # held for all of it
    d = mk([[], [0], [0]], [1, 1, 1], out_bytes=[4, 0, 0], n_dev=3, bw=2,
           lat=[[0, 3, 9], [0, 0, 0], [0, 0, 0]])
    r = _arb(d, [0, 1, 2])
    assert _xt(r) == [(0, 1, 1, 1, 6), (0, 2, 1, 6, 17)]


def test_zero_length_transfers_chain_at_one_instant():
    # empty outputs over zero-latency links take no time: the second transfer
    # from the same sender starts and ends at the same instant as the first
    d = mk([[], [0], [0], [0]], [5, 1, 1, 1], out_bytes=[0, 0, 0, 0], n_dev=4, bw=1, lat=0)
    r = _arb(d, [0, 1, 2, 3])
    assert _xt(r) == [(0, 1, 5, 5, 5), (0, 2, 5, 5, 5), (0, 3, 5, 5, 5)]
    assert r["finish"].tolist() == [5, 6, 6, 6]


def test_receive_buffer_allocated_when_the_transfer_starts():
    # ops 0 and 1 (10 B each) on accelerator 0 send to accelerator 1 one after
    # the other (0 -> 1 busy over [1, 11)).  Op 0's copy there has no listed
    # consumer, so it is released on arrival at 11; op 1's copy is allocated
    # when its transfer starts at 11, not at its intent (2): at most 10 B are
    # ever live on accelerator 1, within a 15 B capacity.
    d = mk([[], [], [0], [1]], [1, 1, 1, 1], out_bytes=[10, 10, 0, 0], n_dev=2, bw=1, lat=0,
           cons=[[], [3], [], []], cap=[100, 15])
    r = _arb(d, [0, 0, 1, 1])
    assert _xt(r) == [(0, 1, 1, 1, 11), (1, 1, 2, 11, 21)]
    assert r["peak"].tolist() == [20, 10] and r["viol_flag"] == 0
    assert r["finish"].tolist() == [1, 2, 12, 22]
    # the source copies stay until their transfers are done: [0, 11) and [1, 21)
    d.cap[:] = [19, 15]
    r = _arb(d, [0, 0, 1, 1])
    assert (r["viol_flag"], r["viol_time"], r["viol_op"], r["viol_dev"]) == (1, 1, 1, 0)


def test_no_competition_equals_pure_latency():
    g = np.random.default_rng(3)
    # everything on one accelerator: no transfer at all
    for seed in range(20):
        d = random_desc(seed, 40, 4, bytes_hi=500)
        place = np.full(40, seed % 4)
        a, b = _arb(d, place), O.simulate(d, row(place))
        assert a["transfers"].shape[0] == 0
        for k in ("ready", "start", "finish", "peak"):
            assert a[k].tolist() == b[k].tolist(), (seed, k)
    # a chain alternating between two accelerators: one transfer at a time
    n = 30
    d = mk([[]] + [[i - 1] for i in range(1, n)], g.integers(1, 9, n).tolist(),
           out_bytes=g.integers(0, 50, n).tolist(), n_dev=2, bw=3, lat=2)
    place = [i % 2 for i in range(n)]
    a, b = _arb(d, place), O.simulate(d, row(place))
    assert a["transfers"].shape[0] == n - 1
    for k in ("ready", "start", "finish", "peak"):
        assert a[k].tolist() == b[k].tolist(), k
    assert a["score"] == b["score"] and a["makespan"] == b["makespan"]


def _rand(seed, n_hi=16, d_hi=4, dur_hi=8):
    g = np.random.default_rng(20_000 + seed)
    n = int(g.integers(1, n_hi))
    D = int(g.integers(1, d_hi + 1))
    d = random_desc(seed, n, D, dur_hi=dur_hi, bytes_hi=40, explicit_cons=bool(seed % 2),
                    link_hetero=bool(seed % 3), n_types=(2 + seed % 2) if seed % 4 == 3 else 0)
    d.bw[:] = np.random.default_rng(seed).integers(2, 20, d.bw.shape[0])
    d.lat[:] = np.random.default_rng(seed + 1).integers(0, 5, d.lat.shape[0])
    if seed % 5 == 0:
        d.out_bytes[::3] = 0
        d.lat[:] = 0               # zero-length transfers
    if seed % 3 == 0:              # links shared by both directions of a pair
        link = np.zeros((D, D), np.int32)
        for a in range(D):
            for b in range(D):
                link[a, b] = min(a, b) * D + max(a, b)
        d.link_id = link.reshape(-1)
    elif seed % 3 == 1 and D > 2:  # accelerators 2m and 2m+1 share one uplink
        d.link_id = np.repeat(np.arange(D, dtype=np.int32) // 2 * D, D)
    place = g.integers(0, D, n)
    return d, place


@pytest.mark.parametrize("block", range(6))
def test_tick_stepped_arbitration_equals_oracle(block):
    for seed in range(block * 40, block * 40 + 40):
        d, place = _rand(seed)
        rd, st, fi, xs = refsim.tick_sim_arb(d, place)
        r = _arb(d, place)
        assert r["ready"].tolist() == rd, seed
        assert r["start"].tolist() == st, seed
        assert r["finish"].tolist() == fi, seed
        assert _xt(r) == [(x["p"], x["e"], x["intent"], x["start"], x["done"]) for x in xs], seed
        want = refsim.summarize(d, place, st, fi, transfers=xs)
        for k in ("viol_flag", "viol_time", "viol_op", "viol_dev", "makespan", "score",
                  "sla_miss", "events"):
            assert r[k] == want[k], (seed, k)
        assert r["peak"].tolist() == want["peak"], seed
        assert r["req_done"].tolist() == want["req_done"], seed


def test_tick_stepped_arbitration_equals_oracle_on_larger_graphs():
    for seed in range(1000, 1040):
        d, place = _rand(seed, n_hi=40, d_hi=6, dur_hi=10)
        rd, st, fi, xs = refsim.tick_sim_arb(d, place)
        r = _arb(d, place)
        assert r["finish"].tolist() == fi and r["start"].tolist() == st and r["ready"].tolist() == rd, seed
        assert _xt(r) == [(x["p"], x["e"], x["intent"], x["start"], x["done"]) for x in xs], seed
        want = refsim.summarize(d, place, st, fi, transfers=xs)
        assert r["peak"].tolist() == want["peak"] and r["viol_time"] == want["viol_time"], seed


def _check_table(d, place, r):
    """Every property the arbitration rule fixes, on one transfer table
    (transfers of nonzero length only)."""
    D = d.n_dev
    dev = [int(x) for x in place]
    xs = _xt(r)
    link = (lambda a, b: a * D + b) if d.link_id is None else (lambda a, b: int(d.link_id[a * D + b]))
    pred, succ, _ = refsim.lists(d)
    fin = r["finish"].tolist()
    # one transfer per (producer, distinct remote accelerator of a successor),
    # raised at the producer's finish, lasting the transfer estimate
    want = sorted((p, e) for p in range(d.n_ops) for e in {dev[j] for j in succ[p]} if e != dev[p])
    assert sorted((p, e) for p, e, *_ in xs) == want
    for p, e, it, st, dn in xs:
        assert it == fin[p] and st >= it
        assert dn - st == refsim.xfer(d, dev[p], e, d.out_bytes[p]) > 0

    def clash(x, y):
        return (dev[x[0]] == dev[y[0]] or x[1] == y[1] or
                link(dev[x[0]], x[1]) == link(dev[y[0]], y[1]))
    order = {(x[0], x[1]): k for k, x in enumerate(xs)}
    instants = sorted({v for x in xs for v in x[2:]})
    for t in instants:
        active = [y for y in xs if y[3] <= t < y[4]]
        # conflict-free
        for a in range(len(active)):
            for b in range(a + 1, len(active)):
                assert not clash(active[a], active[b]), (t, active[a], active[b])
        for x in xs:
            if not (x[2] <= t < x[3]):
                continue
            # a waiting intent is held by an earlier-started or earlier-ordered transfer
            assert any(clash(x, y) and (y[3] < t or order[(y[0], y[1])] < order[(x[0], x[1])])
                       for y in active), (t, x)
    # FIFO per pair
    for x in xs:
        for y in xs:
            if dev[x[0]] == dev[y[0]] and x[1] == y[1] and (x[2], x[0]) < (y[2], y[0]):
                assert x[3] < y[3]


@pytest.mark.parametrize("seed", range(12))
def test_transfer_tables_obey_the_arbitration_rule(seed):
    g = np.random.default_rng(seed)
    D = int(g.integers(2, 9))
    d = random_desc(100 + seed, 150, D, dur_hi=40, bytes_hi=600, n_types=2 if seed % 3 == 0 else 0)
    d.bw[:] = g.integers(5, 60, D * D)
    d.lat[:] = g.integers(1, 8, D * D)      # every transfer takes >= 1 us
    if seed % 2:
        d.link_id = g.integers(0, max(D * D // 3, 1), D * D).astype(np.int32)
    place = g.integers(0, D, 150)
    r = _arb(d, place)
    assert r["status"] == 0
    _check_table(d, place, r)


@pytest.mark.parametrize("seed,D", [(0, 40), (1, 64)])
def test_transfer_tables_obey_the_rule_on_many_accelerators(seed, D):
    """The same rule checks with more accelerators than a warp has lanes
    (the library's wide arbitrated kernel), with pair-shared links."""
    g = np.random.default_rng(200 + seed)
    d = random_desc(300 + seed, 240, D, dur_hi=40, bytes_hi=600)
    d.bw[:] = g.integers(5, 60, D * D)
    d.lat[:] = g.integers(1, 8, D * D)
    a, b = np.meshgrid(np.arange(D), np.arange(D), indexing="ij")
    d.link_id = (np.minimum(a, b) * D + np.maximum(a, b)).astype(np.int32).reshape(-1)
    # few accelerators per op neighbourhood so that transfers compete
    place = g.integers(0, 6, 240) * (D // 6)
    r = _arb(d, place)
    assert r["status"] == 0 and r["transfers"].shape[0] > 50
    _check_table(d, place, r)


def test_rejects_bad_link_ids():
    d = mk([[], [0]], [1, 1], n_dev=2)
    d.link_id = np.array([0, 4, 1, 0], np.int32)   # 4 >= D*D
    assert O.check(d, arbitrated=True) == O.EINVAL
    d.link_id = np.array([9, 1, 2, -3], np.int32)  # the diagonal is not read
    assert O.check(d, arbitrated=True) == 0


def test_incremental_is_the_full_arbitrated_simulation_of_the_moved_placement():
    d = random_desc(5, 80, 4)
    base = np.random.default_rng(1).integers(0, 4, 80).astype(np.uint8)
    mv = W.random_moves(3, 24, base, 4, max_moves=5)
    # two malformed move lists: an out-of-range device and a repeated op
    mv.dev[mv.off[2]] = 9
    assert mv.off[6] - mv.off[5] > 1
    mv.op[mv.off[5] + 1] = mv.op[mv.off[5]]
    s, pk, rq = O.incremental_batch(d, base, mv, arbitrated=True)
    sl, _, _ = O.incremental_batch(d, base, mv)
    assert s["status"].tolist() == sl["status"].tolist() and s["status"][2] == O.SIM_MOVE_RANGE
    assert s["status"][5] == O.SIM_MOVE_DUP
    for k in range(24):
        if s["status"][k]:
            continue
        pl = base.copy()
        a, b = mv.off[k], mv.off[k + 1]
        pl[mv.op[a:b]] = mv.dev[a:b]
        r = _arb(d, pl)
        assert (r["score"], r["makespan"], r["viol_flag"]) == (s["score"][k], s["makespan"][k], s["viol_flag"][k])
        assert r["peak"].tolist() == pk[k].tolist() and s["events"][k] == d.n_ops


# ---------------------------------------------------------------------------
# Resuming arbitrated incremental candidates at T0
# ---------------------------------------------------------------------------

def _inc_helpers():
    import test_oracle_incremental as TI
    return TI._t0, TI._applied


@pytest.mark.parametrize("seed", range(12))
def test_arbitrated_prefix_before_t0_is_unchanged(seed):
    """What resuming an arbitrated candidate at T0 relies on: with T0 taken
    from the arbitrated base's finish times, every op whose arbitrated base
    ready time is < T0 keeps its ready, start and finish times in the moved
    placement's arbitrated schedule, every other op is ready at or after T0,
    and so is every transfer that touches a moved op's predecessors."""
    from paper_2608_15762_gb300.workloads import random_desc, random_moves
    t0f, applied = _inc_helpers()
    g = np.random.default_rng(900 + seed)
    n = int(g.integers(5, 150))
    D = int(g.integers(2, 7))
    d = random_desc(7000 + seed, n, D, explicit_cons=bool(seed % 2), dur_hi=300)
    if seed % 3 == 2:
        d.link_id = np.asarray([(min(s, e) * D + max(s, e)) for s in range(D) for e in range(D)], np.int32)
    base = g.integers(0, D, n).astype(np.uint8)
    mv = random_moves(300 + seed, 30, base, D, max_moves=5, allow_noop=False)
    rb = O.simulate(d, base, arbitrated=True)
    checked = 0
    for k in range(30):
        t0 = t0f(d, base, mv, k, rb["finish"].tolist())
        if t0 is None:
            continue
        rc = O.simulate(d, applied(base, mv, k), arbitrated=True)
        early = rb["ready"] < t0
        assert np.array_equal(rc["ready"][early], rb["ready"][early])
        assert np.array_equal(rc["start"][early], rb["start"][early])
        assert np.array_equal(rc["finish"][early], rb["finish"][early])
        assert (rc["ready"][~early] >= t0).all()
        checked += 1
    assert checked > 0


@pytest.mark.parametrize("seed", range(6))
def test_resumed_event_count(seed):
    """resumed=True changes only `events`: the ops whose arbitrated base ready
    time is >= T0 (0 without an effective move); every other field is the
    moved placement's full arbitrated simulation."""
    from paper_2608_15762_gb300.workloads import random_desc, random_moves
    t0f, _ = _inc_helpers()
    g = np.random.default_rng(60 + seed)
    n = int(g.integers(20, 120))
    D = int(g.integers(2, 6))
    d = random_desc(7100 + seed, n, D, dur_hi=200)
    base = g.integers(0, D, n).astype(np.uint8)
    mv = random_moves(400 + seed, 24, base, D, max_moves=4)
    full, pf, rf = O.incremental_batch(d, base, mv, arbitrated=True)
    res, pr, rr = O.incremental_batch(d, base, mv, arbitrated=True, resumed=True)
    rb = O.simulate(d, base, arbitrated=True)
    for f in full.dtype.names:
        if f not in ("events", "reserved"):
            assert np.array_equal(full[f], res[f]), f
    assert np.array_equal(pf, pr) and np.array_equal(rf, rr)
    assert (full["events"][full["status"] == 0] == n).all()
    for k in range(24):
        if res["status"][k]:
            continue
        t0 = t0f(d, base, mv, k, rb["finish"].tolist())
        want = 0 if t0 is None else int((rb["ready"] >= t0).sum())
        assert res["events"][k] == want
