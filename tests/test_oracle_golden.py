"""Hand-derived worked examples (tests/golden/*.json, each with the passages
it follows and its step-by-step derivation) pin the oracle's arithmetic,
with pure-latency or (transfer_mode 1) arbitrated transfers."""
import glob
import json
import os

import numpy as np
import pytest

from helpers import mk, row
from oracle import oracle as O

FILES = sorted(glob.glob(os.path.join(os.path.dirname(__file__), "golden", "*.json")))


@pytest.mark.parametrize("path", FILES, ids=[os.path.basename(f) for f in FILES])
def test_golden(path):
    with open(path) as f:
        fx = json.load(f)
    g = fx["graph"]
    for case in fx["cases"]:
        d = mk(g["preds"], g["dur"], g["out_bytes"], n_dev=g["n_dev"], bw=g["bw"], lat=g["lat"],
               release=g.get("release"), avail0=g.get("avail0"), req_id=g.get("req_id"),
               deadline=g.get("deadline"), cap=case["cap"])
        arb = g.get("transfer_mode", 0) == 1
        if g.get("link_id") is not None:
            d.link_id = np.asarray(g["link_id"], np.int32)
        r = O.simulate(d, row(fx["place"]), arbitrated=arb)
        if "transfers" in case:
            assert r["transfers"].tolist() == case["transfers"]
        assert r["ready"].tolist() == case["ready"]
        assert r["start"].tolist() == case["start"]
        assert r["finish"].tolist() == case["finish"]
        assert r["peak"].tolist() == case["peak"]
        viol = None if not r["viol_flag"] else [r["viol_time"], r["viol_op"], r["viol_dev"]]
        assert viol == case["viol"]
        assert r["makespan"] == case["makespan"]
        assert r["score"] == case["score"]
        assert r["sla_miss"] == case["sla_miss"]
        assert r["req_done"].tolist() == case["req_done"]
