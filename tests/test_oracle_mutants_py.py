"""Plant plausible mistakes in scratch copies of the round and estimator
oracles (on the CPU) and check that their pins catch every one: ties to the
larger op id, first-in-first-out collection, admission that ignores the
batch, a strict budget test, a frontier of done predecessors only, wrapping
partition slots, a cap that ignores issued ops; fitting the last batch only,
floor for rint, a zero lower clamp, an uninverted bandwidth, fitting
rank-deficient data, using unfitted estimators."""
import importlib
import inspect
import os
import types

import pytest

import test_oracle_estimators as TE
import test_oracle_round as TR

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

ROUND_MUTANTS = {
    "ties_to_larger_id": [("key=lambda i: (int(prio[i]), i))", "key=lambda i: (int(prio[i]), -i))")],
    "fifo_collection": [("x = heapq.heappop(heap)", "x = heap.pop(0)"), ("heapq.heappush(heap, j)", "heap.append(j)")],
    "admission_ignores_batch": [("all(state[p] != 0 or p in marked for p in pred[j])",
                                 "all(state[p] != 0 for p in pred[j])")],
    "strict_budget": [("if issued >= budget:", "if issued > budget:")],
    "frontier_done_only": [("state[i] == 0 and all(state[p] != 0 for p in pred[i])",
                            "state[i] == 0 and all(state[p] == 2 for p in pred[i])")],
    "wrapping_slots": [("rows[p, x] = part_dev[part_off[p] + s] if 0 <= s < size else 255",
                        "rows[p, x] = part_dev[part_off[p] + s % size]")],
    "cap_ignores_issued": [("cap = min(max_batch, budget - issued)", "cap = max_batch")],
}

EST_MUTANTS = {
    "last_batch_only": [("self.xs[e] = np.vstack([self.xs[e], x[a:b]])", "self.xs[e] = x[a:b].copy()"),
                        ("self.ys[e] = np.concatenate([self.ys[e], y[a:b]])", "self.ys[e] = y[a:b].copy()")],
    "floor_for_rint": [("r = np.rint(v)", "r = np.floor(v)")],
    "zero_lower_clamp": [("out[i, t] = clamp_rint(float(np.dot(beta[e], x[i])), 1)",
                          "out[i, t] = clamp_rint(float(np.dot(beta[e], x[i])), 0)")],
    "uninverted_bandwidth": [("bw[q] = clamp_rint(1.0 / alpha, 1) if alpha > 0 else MAX_TICKS",
                              "bw[q] = clamp_rint(alpha, 1) if alpha > 0 else MAX_TICKS")],
    "rank_ignored": [(" and np.linalg.matrix_rank(X) == self.n_feat", "")],
    "unfitted_used": [("if e < 0 or not fitted[e]:", "if e < 0:")],
}


def _mutant(modname, edits):
    path = os.path.join(ROOT, "oracle", modname + ".py")
    src = open(path).read()
    for old, new in edits:
        assert src.count(old) == 1, (modname, old)
        src = src.replace(old, new)
    mod = types.ModuleType("mutant_" + modname)
    mod.__file__ = path
    exec(compile(src, path, "exec"), mod.__dict__)
    return mod


def _pins_fail(test_mod, attr, mutant):
    """True if at least one pin of test_mod fails with its oracle replaced."""
    saved = getattr(test_mod, attr)
    setattr(test_mod, attr, mutant)
    try:
        for name, fn in inspect.getmembers(test_mod, inspect.isfunction):
            if not name.startswith("test_"):
                continue
            params = getattr(fn, "pytestmark", [])
            cases = [()]
            for m in params:
                if m.name == "parametrize":
                    cases = [(v,) for v in m.args[1]]
            for c in cases:
                try:
                    fn(*c)
                except AssertionError:
                    return True
        return False
    finally:
        setattr(test_mod, attr, saved)


@pytest.mark.parametrize("name", sorted(ROUND_MUTANTS))
def test_round_pins_catch(name):
    assert _pins_fail(TR, "R", _mutant("round", ROUND_MUTANTS[name])), name


@pytest.mark.parametrize("name", sorted(EST_MUTANTS))
def test_estimator_pins_catch(name):
    assert _pins_fail(TE, "E", _mutant("estimators", EST_MUTANTS[name])), name


def test_unmutated_oracles_pass_their_pins():
    assert not _pins_fail(TR, "R", importlib.import_module("oracle.round"))
    assert not _pins_fail(TE, "E", importlib.import_module("oracle.estimators"))
