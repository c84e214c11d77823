"""GPU parity on structured placements (each request's ops in contiguous
stages on random accelerators, like the pre-defined partitions of Sec.
3.4.2): few cross-accelerator transfers and long same-accelerator runs, the
opposite regime of uniform i.i.d. placements.  Every candidate of the
prefill and two-type prefill workloads, with pure-latency and with
arbitrated transfers, bit for bit against the oracle."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

from gpu_common import compare, torch_place  # noqa: E402
from oracle import oracle as O  # noqa: E402
from paper_2608_15762_gb300 import gmgsim as G  # noqa: E402
from paper_2608_15762_gb300 import workloads as W  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2608_15762_gb300 import build
    build.build()
    assert torch.cuda.is_available()


@pytest.mark.parametrize("cfg", [2, 6])
@pytest.mark.parametrize("arbitrated", [False, True])
def test_structured_placements_every_candidate(cfg, arbitrated):
    wl = W.make_workload(cfg)
    rows = wl.structured_full_rows(range(wl.n_full))
    g = G.gmg_create(wl.desc)
    out = G.sim_batch(g, torch_place(rows), req_done=True, arbitrated=arbitrated)
    best = G.select_best(out)
    torch.cuda.synchronize()
    s, pk, rq = O.simulate_batch(wl.desc, rows, arbitrated=arbitrated)
    compare(out.to_numpy(), s, pk, rq)
    assert best.cpu().tolist() == list(O.select_best(s, 0))
    assert (s["status"] == 0).all()
