"""Shared helpers of the GPU tests: run the CUDA path and the oracle on the
same seeded inputs and compare every output field bit for bit."""
import numpy as np

from oracle import oracle as O

FIELDS = ("status", "viol_flag", "viol_op", "viol_dev", "viol_time", "makespan", "score", "events",
          "sla_miss")


def torch_place(rows, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(rows)).to(device)


def compare(gpu: dict, summ, peak, req=None, ks=None, check_events=True):
    """gpu: SimOut.to_numpy(); summ/peak/req: oracle arrays for candidates ks
    (all if None)."""
    ks = np.arange(summ.shape[0]) if ks is None else np.asarray(ks)
    for f in FIELDS:
        if f == "events" and not check_events:
            continue
        got = gpu[f][ks] if ks is not None else gpu[f]
        want = summ[f] if len(summ) == len(ks) else summ[f][ks]
        bad = np.flatnonzero(got != want)
        assert bad.size == 0, "field %s differs at candidates %s: gpu %s oracle %s" % (
            f, ks[bad[:5]], got[bad[:5]], want[bad[:5]])
    gp = gpu["peak"][ks]
    bad = np.flatnonzero((gp != peak).any(axis=1))
    assert bad.size == 0, "peak differs at candidates %s" % ks[bad[:5]]
    if req is not None and gpu.get("req_done") is not None:
        gr = gpu["req_done"][ks]
        bad = np.flatnonzero((gr != req).any(axis=1)) if req.size else np.zeros(0, int)
        assert bad.size == 0, "req_done differs at candidates %s" % ks[bad[:5]]


def oracle_rows(desc, rows, nthreads=0):
    return O.simulate_batch(desc, rows, nthreads=nthreads)
