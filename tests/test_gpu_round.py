"""GPU parity of the scheduling round (include/gmground.h) against the round
oracle: frontier counts, the chosen op, the batch in collection order, the
candidate rows, the winning partition and the written-back state and
placement, exactly, over several consecutive rounds."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import round as R  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


def _closed_states(g, desc, p_sched):
    pred, _ = R._lists(desc)
    st = np.zeros(desc.n_ops, np.uint8)
    for i in range(desc.n_ops):
        if all(st[q] != 0 for q in pred[i]) and g.random() < p_sched:
            st[i] = 2 if g.random() < 0.6 else 1
    return st


def _dev(a, dt):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=dt)).cuda()


def _run_rounds(desc, g, n_rounds, n_tmpl, n_roles, part_off, part_dev, budget, max_batch, p_sched, D):
    n = desc.n_ops
    ld = W.placement_ld(n)
    state = _closed_states(g, desc, p_sched)
    place = np.zeros(ld, np.uint8)
    place[:n] = g.integers(0, D, n)
    prio = g.integers(0, 1000, n)
    tmpl = g.integers(0, n_tmpl, n).astype(np.int32)
    role = g.integers(0, n_roles, n).astype(np.int32)
    n_part = len(part_off) - 1
    sizes = np.diff(part_off)
    mapping = np.zeros((n_tmpl, n_part, n_roles), np.int32)
    for p in range(n_part):
        mapping[:, p, :] = g.integers(0, sizes[p] + (1 if p == n_part - 1 else 0), (n_tmpl, n_roles))
    mapping = mapping.reshape(-1)
    gm = G.gmg_create(desc)
    st_d, pl_d = _dev(state, np.uint8), _dev(place, np.uint8)
    rnd = G.Round(gm, st_d, pl_d, _dev(prio, np.int64), _dev(tmpl, np.int32), _dev(role, np.int32),
                  _dev(part_off, np.int32), _dev(part_dev, np.uint8), _dev(mapping, np.int32), n_roles,
                  budget, max_batch)
    statuses = []
    for r in range(n_rounds):
        info, batch, rows, best, state, place = R.round_step(desc, state, place, prio, tmpl, role, part_off,
                                                             part_dev, mapping, n_roles, budget, max_batch)
        rnd.step()
        torch.cuda.synchronize()
        gi = rnd.info.cpu().numpy().tolist()
        assert gi == info, (r, gi, info)
        nb = info[0]
        assert rnd.batch[:nb].cpu().numpy().tolist() == batch, r
        if info[5] in (R.BATCH, R.NO_FEASIBLE):
            assert np.array_equal(rnd.rows.cpu().numpy()[:, :n], rows[:, :n]), r
            assert rnd.best.cpu().numpy().tolist() == list(best), r
        assert np.array_equal(st_d.cpu().numpy(), state), r
        assert np.array_equal(pl_d.cpu().numpy(), place), r
        statuses.append(info[5])
        # the executor finishes some issued ops between rounds
        fin = (state == 1) & (g.random(n) < 0.5)
        state[fin] = 2
        st_d.copy_(_dev(state, np.uint8))
    return statuses


@pytest.mark.parametrize("seed", range(4))
def test_random_graphs_several_rounds(seed):
    g = np.random.default_rng(seed)
    D = 5
    desc = W.random_desc(400 + seed, 300, D, dur_hi=80, edge_p=0.6, cap=1 << 40)
    part_off = [0, 1, 2, 4, 5, 8]
    part_dev = [0, 4, 1, 2, 3, 0, 1, 2]
    st = _run_rounds(desc, g, 8, n_tmpl=3, n_roles=4, part_off=part_off, part_dev=part_dev, budget=60,
                     max_batch=16, p_sched=0.3, D=D)
    assert R.BATCH in st


def test_budget_and_empty_rounds():
    g = np.random.default_rng(9)
    desc = W.random_desc(9, 60, 3, dur_hi=30)
    st = _run_rounds(desc, g, 12, n_tmpl=1, n_roles=2, part_off=[0, 1, 2, 3], part_dev=[0, 1, 2], budget=6,
                     max_batch=4, p_sched=0.5, D=3)
    assert R.BUDGET in st or R.EMPTY in st or R.NO_FEASIBLE in st


def test_prefill_requests_with_layer_partitions():
    """The prefill graph (8 requests x 32 layers): one template, role = op
    position in the request, partitions of 1, 2 and 4 accelerators, a
    request's layers split evenly over a partition's accelerators."""
    g = np.random.default_rng(11)
    wl = W.config2()
    desc = wl.desc
    per = desc.n_ops // 8
    part_off = [0, 1, 2, 3, 4, 5, 6, 7, 8, 10, 12, 14, 16, 20, 24]
    part_dev = list(range(8)) + [0, 1, 2, 3, 4, 5, 6, 7] + [0, 1, 2, 3, 4, 5, 6, 7]
    n_part = len(part_off) - 1
    sizes = np.diff(part_off)
    mapping = np.zeros((1, n_part, per), np.int32)
    for p in range(n_part):
        mapping[0, p, :] = np.arange(per) * sizes[p] // per
    n = desc.n_ops
    ld = W.placement_ld(n)
    state = np.zeros(n, np.uint8)
    place = np.zeros(ld, np.uint8)
    place[:n] = g.integers(0, 8, n)
    prio = np.repeat(desc.deadline, per)
    tmpl = np.zeros(n, np.int32)
    role = np.tile(np.arange(per), 8).astype(np.int32)
    gm = G.gmg_create(desc)
    st_d, pl_d = _dev(state, np.uint8), _dev(place, np.uint8)
    rnd = G.Round(gm, st_d, pl_d, _dev(prio, np.int64), _dev(tmpl, np.int32), _dev(role, np.int32),
                  _dev(part_off, np.int32), _dev(np.array(part_dev), np.uint8), _dev(mapping.reshape(-1), np.int32),
                  per, budget=128, max_batch=64)
    for r in range(4):
        info, batch, rows, best, state, place = R.round_step(desc, state, place, prio, tmpl, role, part_off,
                                                             part_dev, mapping.reshape(-1), per, 128, 64)
        rnd.step()
        torch.cuda.synchronize()
        assert rnd.info.cpu().numpy().tolist() == info
        assert rnd.batch[:info[0]].cpu().numpy().tolist() == batch
        assert rnd.best.cpu().numpy().tolist() == list(best)
        assert np.array_equal(st_d.cpu().numpy(), state) and np.array_equal(pl_d.cpu().numpy(), place)
        state[state == 1] = 2
        st_d.copy_(_dev(state, np.uint8))


def _one_round(desc, state, place, budget, max_batch, part_off, part_dev, mapping, n_roles, prio=None):
    n = desc.n_ops
    prio = np.arange(n) if prio is None else prio
    tmpl, role = np.zeros(max(n, 1), np.int32), np.zeros(max(n, 1), np.int32)
    gm = G.gmg_create(desc)
    st_d, pl_d = _dev(np.asarray(state, np.uint8) if n else np.zeros(1, np.uint8), np.uint8), _dev(place, np.uint8)
    rnd = G.Round(gm, st_d, pl_d, _dev(prio if n else np.zeros(1), np.int64), _dev(tmpl, np.int32),
                  _dev(role, np.int32), _dev(part_off, np.int32), _dev(part_dev, np.uint8), _dev(mapping, np.int32),
                  n_roles, budget, max_batch)
    rnd.step()
    torch.cuda.synchronize()
    want = R.round_step(desc, state, place, prio, tmpl, role, part_off, part_dev, mapping, n_roles, budget, max_batch)
    return rnd, st_d, pl_d, want


def test_degenerate_rounds():
    from helpers import mk
    chain = mk([[], [0], [1], [2]], [3, 4, 5, 6], n_dev=2, bw=1, lat=1)
    place = np.zeros(16, np.uint8)
    args = dict(part_off=[0, 1, 2], part_dev=[0, 1], mapping=[0, 0], n_roles=1)
    # everything done: the unscheduled frontier is empty
    rnd, st, pl, want = _one_round(chain, [2, 2, 2, 2], place, 8, 8, **args)
    assert rnd.info.cpu().tolist() == want[0] and want[0][5] == R.EMPTY
    # budget 0: nothing is scheduled even with a frontier
    rnd, st, pl, want = _one_round(chain, [0, 0, 0, 0], place, 0, 8, **args)
    assert rnd.info.cpu().tolist() == want[0] and want[0][5] == R.BUDGET
    assert st.cpu().tolist() == [0, 0, 0, 0]
    # batch cap 1: exactly the chosen op
    rnd, st, pl, want = _one_round(chain, [0, 0, 0, 0], place, 8, 1, **args)
    assert rnd.info.cpu().tolist() == want[0] and want[1] == [0]
    assert st.cpu().tolist() == want[4].tolist() and pl.cpu().tolist() == want[5].tolist()
    # every candidate maps to a slot outside its partition: nothing feasible, nothing written
    bad = dict(part_off=[0, 1, 2], part_dev=[0, 1], mapping=[3, 3], n_roles=1)
    rnd, st, pl, want = _one_round(chain, [0, 0, 0, 0], place, 8, 8, **bad)
    assert want[0][5] == R.NO_FEASIBLE and rnd.info.cpu().tolist() == want[0]
    assert st.cpu().tolist() == [0, 0, 0, 0] and pl.cpu().tolist() == place.tolist()
    # an empty graph
    empty = mk([], [], n_dev=2)
    rnd, st, pl, want = _one_round(empty, np.zeros(0, np.uint8), place, 8, 8, **args)
    assert rnd.info.cpu().tolist()[5] == R.EMPTY and rnd.info.cpu().tolist()[1] == -1
