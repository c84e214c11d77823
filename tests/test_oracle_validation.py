"""The oracle rejects malformed graphs (host-side validation rules)."""
import numpy as np

from helpers import mk
from oracle import oracle as O


def _ok():
    return mk([[], [0], [0, 1]], [3, 4, 5], [1, 2, 3], n_dev=2, bw=2, lat=1)


def test_valid_graph_passes():
    assert O.check(_ok()) == 0


def test_rejections():
    d = _ok(); d.dur[1] = 0
    assert O.check(d) == O.EINVAL
    d = _ok(); d.out_bytes[0] = -1
    assert O.check(d) == O.EINVAL
    d = _ok(); d.release[2] = -5
    assert O.check(d) == O.EINVAL
    d = _ok(); d.pred_idx[0] = 1     # op 1 depends on itself
    assert O.check(d) == O.ENOTTOPO
    d = _ok(); d.pred_idx[0] = 2     # op 1 depends on a later op
    assert O.check(d) == O.ENOTTOPO
    d = _ok(); d.pred_idx[1] = 1; d.pred_idx[2] = 1   # duplicate predecessor of op 2
    assert O.check(d) == O.EINVAL
    d = _ok(); d.bw[1] = 0
    assert O.check(d) == O.EINVAL
    d = _ok(); d.lat[2] = -1
    assert O.check(d) == O.EINVAL
    d = _ok(); d.base[:] = [5, 0]; d.cap[:] = [4, 10]
    assert O.check(d) == O.EINVAL
    d = _ok(); d.dur[0] = 1 << 62
    assert O.check(d) == O.ERANGE
    d = _ok(); d.pred_off[1] = 3      # offsets not monotone
    assert O.check(d) == O.EINVAL


def test_consumer_lists_must_be_successors():
    ok = mk([[], [0], [0, 1]], [3, 4, 5], n_dev=2, cons=[[2], [2], []])
    assert O.check(ok) == 0
    bad = mk([[], [0], [1]], [3, 4, 5], n_dev=2, cons=[[2], [], []])
    assert O.check(bad) == O.EINVAL
    dup = mk([[], [0], [0, 1]], [3, 4, 5], n_dev=2, cons=[[2, 2], [], []])
    assert O.check(dup) == O.EINVAL


def test_device_count_limits():
    d = _ok(); d.n_dev = 0
    assert O.check(d) == O.EINVAL
    d = mk([[]], [1], n_dev=256)
    assert O.check(d) == 0
