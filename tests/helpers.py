"""Small hand-built graphs for the tests."""
from __future__ import annotations

import numpy as np

from paper_2608_15762_gb300.workloads import GmgDesc, INT64_MAX


def mk(preds, dur, out_bytes=None, n_dev=2, release=None, req_id=None, scored=None,
       deadline=None, cap=None, base=None, avail0=None, bw=1, lat=0, cons=None) -> GmgDesc:
    """Build a GmgDesc from python lists.  ``bw``/``lat`` may be scalars
    (uniform off-diagonal) or D x D nested lists."""
    n = len(preds)
    pred_off = np.zeros(n + 1, np.int32)
    pred_off[1:] = np.cumsum([len(p) for p in preds])
    pred_idx = np.array([q for p in preds for q in p], np.int32)
    D = n_dev
    if np.isscalar(bw):
        bw = np.full(D * D, bw, np.int64)
    if np.isscalar(lat):
        lat = np.full(D * D, lat, np.int64)
    n_req = 0 if deadline is None else len(deadline)
    cons_off = cons_idx = None
    if cons is not None:
        cons_off = np.zeros(n + 1, np.int32)
        cons_off[1:] = np.cumsum([len(c) for c in cons])
        cons_idx = np.array([c for cs in cons for c in cs], np.int32)
    return GmgDesc(
        n_dev=D, pred_off=pred_off, pred_idx=pred_idx,
        dur=np.asarray(dur, np.int64),
        out_bytes=np.zeros(n, np.int64) if out_bytes is None else np.asarray(out_bytes, np.int64),
        release=np.zeros(n, np.int64) if release is None else np.asarray(release, np.int64),
        req_id=np.full(n, -1, np.int32) if req_id is None else np.asarray(req_id, np.int32),
        scored=np.ones(n, np.uint8) if scored is None else np.asarray(scored, np.uint8),
        deadline=np.zeros(0, np.int64) if deadline is None else np.asarray(deadline, np.int64),
        cap=np.full(D, INT64_MAX, np.int64) if cap is None else np.asarray(cap, np.int64),
        base=np.zeros(D, np.int64) if base is None else np.asarray(base, np.int64),
        avail0=np.zeros(D, np.int64) if avail0 is None else np.asarray(avail0, np.int64),
        bw=np.asarray(bw, np.int64).reshape(-1), lat=np.asarray(lat, np.int64).reshape(-1),
        cons_off=cons_off, cons_idx=cons_idx).normalized()


def row(place, ld=None):
    place = list(place)
    ld = ld or max(16, (len(place) + 15) // 16 * 16)
    r = np.zeros(ld, np.uint8)
    r[:len(place)] = place
    return r


def summary_dict(s):
    return {k: int(s[k]) for k in s.dtype.names if k != "reserved"}
