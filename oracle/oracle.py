"""ctypes wrapper of the CPU oracle (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this module.  It loads ``liboracle_sim.so`` (built by
``oracle/build.py``) and exposes numpy-level calls:

* ``check(desc)`` -> 0 or a negative error code,
* ``simulate(desc, place_row, arbitrated=False)`` -> dict with summary
  fields, peak, req_done, ready/start/finish per op (arbitrated: transfers
  through the arbiter of Sec. 3.5.2, plus the transfer table),
* ``transfers(desc, place_row)`` -> the arbitrated transfers of one placement,
* ``simulate_batch(desc, place, nthreads)`` -> structured summaries, peaks,
  req_done,
* ``incremental_batch(desc, base, moves, nthreads)`` -> same,
* ``select_best(summary, mode)`` -> (best_k, best_score).
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from . import build as _build

SUMMARY_DTYPE = np.dtype([
    ("status", np.int32), ("viol_flag", np.int32), ("viol_op", np.int32),
    ("viol_dev", np.int32), ("viol_time", np.int64), ("makespan", np.int64),
    ("score", np.int64), ("events", np.int64), ("sla_miss", np.int32),
    ("reserved", np.int32)])
assert SUMMARY_DTYPE.itemsize == 56

SIM_OK, SIM_BADDEV, SIM_MOVE_RANGE, SIM_MOVE_DUP, SIM_BADBASE = 0, 1, 2, 3, 4
EINVAL, ENOTTOPO, ERANGE = -1, -2, -3


class _Graph(C.Structure):
    _fields_ = [("n_ops", C.c_int32), ("n_edges", C.c_int32), ("n_dev", C.c_int32),
                ("n_req", C.c_int32)] + [
        (name, C.c_void_p) for name in (
            "pred_off", "pred_idx", "cons_off", "cons_idx", "dur", "out_bytes", "release",
            "req_id", "scored", "deadline", "cap", "base", "avail0", "bw", "lat")] + [
        ("n_types", C.c_int32), ("dev_type", C.c_void_p), ("dur_type", C.c_void_p),
        ("transfer_mode", C.c_int32), ("link_id", C.c_void_p)]


_LIB = None


def lib():
    global _LIB
    if _LIB is None:
        path = os.environ.get("ORACLE_LIB_OVERRIDE") or _build.build()
        L = C.CDLL(path)
        vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
        L.orc_check.argtypes = [vp]
        L.orc_check.restype = C.c_int
        L.orc_hw_threads.restype = i32
        L.orc_simulate.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp]
        L.orc_simulate.restype = C.c_int
        L.orc_simulate_batch.argtypes = [vp, vp, i64, i32, i32, vp, vp, vp]
        L.orc_simulate_batch.restype = C.c_int
        L.orc_incremental_batch.argtypes = [vp, vp, vp, vp, vp, i32, i32, vp, vp, vp, i32]
        L.orc_incremental_batch.restype = C.c_int
        L.orc_select_best.argtypes = [vp, i32, i32, vp]
        L.orc_select_best.restype = i64
        L.orc_transfers.argtypes = [vp, vp, vp, i64]
        L.orc_transfers.restype = i64
        _LIB = L
    return _LIB


def _ptr(a):
    return None if a is None else a.ctypes.data


class _GraphHolder:
    """Keeps the numpy arrays alive while the C struct points into them."""

    def __init__(self, desc, arbitrated=False):
        d = desc.normalized()
        self.desc = d
        self.g = _Graph(d.n_ops, d.n_edges, d.n_dev, d.n_req,
                        _ptr(d.pred_off), _ptr(d.pred_idx), _ptr(d.cons_off), _ptr(d.cons_idx),
                        _ptr(d.dur), _ptr(d.out_bytes), _ptr(d.release), _ptr(d.req_id),
                        _ptr(d.scored), _ptr(d.deadline), _ptr(d.cap), _ptr(d.base),
                        _ptr(d.avail0), _ptr(d.bw), _ptr(d.lat), d.n_types, _ptr(d.dev_type),
                        _ptr(d.dur_by_type), 1 if arbitrated else 0, _ptr(d.link_id))

    @property
    def ref(self):
        return C.byref(self.g)


def hw_threads() -> int:
    return int(lib().orc_hw_threads())


def check(desc, arbitrated=False) -> int:
    h = _GraphHolder(desc, arbitrated)
    return int(lib().orc_check(C.addressof(h.g)))


def simulate(desc, place_row, arbitrated=False) -> dict:
    """One placement; ``arbitrated``: transfers go through the arbiter of
    Sec. 3.5.2 (the dict then also holds ``transfers``)."""
    h = _GraphHolder(desc, arbitrated)
    d = h.desc
    row = np.ascontiguousarray(place_row, dtype=np.uint8)
    assert row.shape[0] >= d.n_ops
    s = np.zeros(1, SUMMARY_DTYPE)
    peak = np.zeros(d.n_dev, np.int64)
    req = np.zeros(max(d.n_req, 1), np.int64)
    r = np.zeros(max(d.n_ops, 1), np.int64)
    st = np.zeros_like(r)
    fi = np.zeros_like(r)
    rc = lib().orc_simulate(C.addressof(h.g), row.ctypes.data, s.ctypes.data, peak.ctypes.data,
                            req.ctypes.data, r.ctypes.data, st.ctypes.data, fi.ctypes.data)
    if rc:
        raise ValueError("oracle rejected the graph: %d" % rc)
    out = {k: s[0][k].item() for k in SUMMARY_DTYPE.names if k != "reserved"}
    out.update(peak=peak, req_done=req[:d.n_req], ready=r[:d.n_ops], start=st[:d.n_ops],
               finish=fi[:d.n_ops])
    if arbitrated:
        out["transfers"] = transfers(desc, row)
    return out


def transfers(desc, place_row) -> np.ndarray:
    """Arbitrated transfers of one placement in arbitration order: int64 rows
    (producer, destination, intent time, start, completion)."""
    h = _GraphHolder(desc, True)
    row = np.ascontiguousarray(place_row, dtype=np.uint8)
    m = lib().orc_transfers(C.addressof(h.g), row.ctypes.data, None, 0)
    if m < 0:
        raise ValueError("oracle rejected the graph: %d" % m)
    rows = np.zeros((max(m, 1), 5), np.int64)
    lib().orc_transfers(C.addressof(h.g), row.ctypes.data, rows.ctypes.data, m)
    return rows[:m]


def simulate_batch(desc, place, nthreads: int = 0, arbitrated=False):
    """place: uint8 [K, ld].  Returns (summary[K], peak[K, D], req_done[K, R])."""
    h = _GraphHolder(desc, arbitrated)
    d = h.desc
    place = np.ascontiguousarray(place, dtype=np.uint8)
    K, ld = place.shape
    s = np.zeros(K, SUMMARY_DTYPE)
    peak = np.zeros((K, d.n_dev), np.int64)
    req = np.zeros((K, max(d.n_req, 1)), np.int64)
    nt = nthreads or hw_threads()
    rc = lib().orc_simulate_batch(C.addressof(h.g), place.ctypes.data, ld, K, nt, s.ctypes.data,
                                  peak.ctypes.data, req.ctypes.data if d.n_req else None)
    if rc:
        raise ValueError("oracle rejected the graph: %d" % rc)
    return s, peak, req[:, :d.n_req]


def incremental_batch(desc, base_place, moves, nthreads: int = 0, arbitrated=False, resumed=False):
    """Move lists against a base placement.  Results are the simulation of
    each moved placement; with arbitrated transfers `resumed` selects what
    `events` counts: False -- every op (the moved placement simulated in
    full); True -- the ops whose arbitrated base ready time is >= T0."""
    h = _GraphHolder(desc, arbitrated)
    d = h.desc
    base = np.ascontiguousarray(base_place, dtype=np.uint8)
    off = np.ascontiguousarray(moves.off, dtype=np.int32)
    op = np.ascontiguousarray(moves.op, dtype=np.int32)
    dv = np.ascontiguousarray(moves.dev, dtype=np.uint8)
    K = off.shape[0] - 1
    s = np.zeros(K, SUMMARY_DTYPE)
    peak = np.zeros((K, d.n_dev), np.int64)
    req = np.zeros((K, max(d.n_req, 1)), np.int64)
    nt = nthreads or hw_threads()
    rc = lib().orc_incremental_batch(C.addressof(h.g), base.ctypes.data, off.ctypes.data,
                                     op.ctypes.data if op.size else None,
                                     dv.ctypes.data if dv.size else None, K, nt, s.ctypes.data,
                                     peak.ctypes.data, req.ctypes.data if d.n_req else None,
                                     1 if resumed else 0)
    if rc:
        raise ValueError("oracle rejected the input: %d" % rc)
    return s, peak, req[:, :d.n_req]


def select_best(summary, mode: int = 0):
    s = np.ascontiguousarray(summary, dtype=SUMMARY_DTYPE)
    best = C.c_int64(0)
    k = lib().orc_select_best(s.ctypes.data, s.shape[0], mode, C.addressof(best))
    return int(k), int(best.value)
