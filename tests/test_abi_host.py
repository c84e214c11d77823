"""The C-ABI library loads, exports every declared symbol, and its host-side
logic (validation, sizing, the exact link division) behaves; no GPU needed."""
import os
import re

import numpy as np
import pytest

from helpers import mk
from paper_2608_15762_gb300 import build, gmgsim as G
from paper_2608_15762_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    build.build()


def test_exports_every_declared_symbol():
    hdr = "".join(open(os.path.join(ROOT, "include", f)).read()
                  for f in sorted(os.listdir(os.path.join(ROOT, "include"))) if f.endswith(".h"))
    names = set(re.findall(r"^\s*(?:[\w\*\s]+?)\b(\w+)\s*\(", hdr, re.M)) - {"if", "sizeof"}
    decl = {n for n in names if n.startswith(("gmg_", "sim_", "base_", "inc_", "select_", "est_", "round_"))}
    assert decl == set(G.EXPORTED), decl ^ set(G.EXPORTED)
    L = G.lib()
    for n in decl:
        assert hasattr(L, n), n


def test_strerror():
    assert G.strerror(0) == "ok"
    assert "topological" in G.strerror(G.GMG_ENOTTOPO) or "predecessor" in G.strerror(G.GMG_ENOTTOPO)
    assert "twice" in G.strerror(G.SIM_MOVE_DUP)


def test_ceil_div_is_exact():
    g = np.random.default_rng(0)
    cases = [(0, 1), (1, 1), (5, 2), (2 ** 53 - 1, 1), (2 ** 53 - 1, 3), (2 ** 53 - 1, 2 ** 61 + 7),
             (12345, 2 ** 40), (2 ** 28, 400000), (2 ** 28 + 1, 50000)]
    for _ in range(3000):
        n = int(g.integers(0, 2 ** 53))
        d = int(g.integers(1, 2 ** int(g.integers(1, 62))))
        cases.append((n, d))
    for n, d in cases:
        assert G.ceil_div_host(n, d) == -(-n // d), (n, d)


def test_workspace_sizing():
    d = W.config1().desc
    assert G.gmg_workspace_bytes(d) > 64 * d.n_ops
    bad = mk([[], [0]], [0, 1])
    assert G.gmg_workspace_bytes(bad) == 0


def _create_rc(desc):
    """gmg_create on a description that fails validation: the library
    rejects it before touching the device (the workspace pointer is never
    dereferenced)."""
    import ctypes as C
    h = G._DescHolder(desc)
    out = C.c_void_p()
    return G.lib().gmg_create(C.addressof(h.c), 256, 1 << 20, None, C.addressof(out))


def test_validation_codes():
    ok = mk([[], [0], [0, 1]], [3, 4, 5], [1, 2, 3], n_dev=2, bw=2, lat=1)
    d = mk([[], [0], [0, 1]], [3, 0, 5], n_dev=2)
    assert _create_rc(d) == G.GMG_EINVAL
    d = mk([[], [1], [0, 1]], [3, 4, 5], n_dev=2)
    assert _create_rc(d) == G.GMG_ENOTTOPO
    d = mk([[], [0], [1, 1]], [3, 4, 5], n_dev=2)
    assert _create_rc(d) == G.GMG_EINVAL
    d = mk([[], [0], [0, 1]], [3, 4, 5], n_dev=2, bw=0)
    assert _create_rc(d) == G.GMG_EINVAL
    d = mk([[], [0], [0, 1]], [3, 4, 5], n_dev=2, cap=[1, 1], base=[2, 0])
    assert _create_rc(d) == G.GMG_EINVAL
    d = mk([[], [0], [0, 1]], [3, 4, 5], n_dev=2, cons=[[2], [0], []])
    assert _create_rc(d) == G.GMG_EINVAL
    d = mk([[], [0], [0, 1]], [1 << 61, 4, 5], n_dev=2)
    assert _create_rc(d) == G.GMG_ERANGE
    d = mk([[], [0], [0, 1]], [3, 4, 5], [1 << 53, 0, 0], n_dev=2)
    assert _create_rc(d) == G.GMG_ERANGE
    d = mk([[]], [1], n_dev=257)
    assert _create_rc(d) == G.GMG_EINVAL
    assert G.gmg_workspace_bytes(ok) > 0


def test_accelerator_type_validation():
    import dataclasses
    base = mk([[], [0], [0, 1]], [3, 4, 5], [1, 2, 3], n_dev=2, bw=2, lat=1)

    def typed(dev_type, table):
        return dataclasses.replace(base, dev_type=np.asarray(dev_type, np.uint8),
                                   dur_by_type=np.asarray(table, np.int64)).normalized()
    assert G.gmg_workspace_bytes(typed([0, 1], [[1, 2], [3, 4], [5, 6]])) > 0
    assert _create_rc(typed([0, 2], [[1, 2], [3, 4], [5, 6]])) == G.GMG_EINVAL   # type >= T
    assert _create_rc(typed([0, 1], [[1, 2], [3, 0], [5, 6]])) == G.GMG_EINVAL   # duration < 1
    assert _create_rc(typed([0, 1], [[1, 2], [1 << 61, 4], [5, 6]])) == G.GMG_ERANGE


def test_link_id_validation_and_option_layout():
    import ctypes as C
    import dataclasses
    base = mk([[], [0], [0, 1]], [3, 4, 5], [1, 2, 3], n_dev=2, bw=2, lat=1)

    def linked(ids):
        return dataclasses.replace(base, link_id=np.asarray(ids, np.int32)).normalized()
    assert G.gmg_workspace_bytes(linked([0, 1, 1, 0])) > 0      # both directions share link 1
    assert G.gmg_workspace_bytes(linked([-7, 3, 2, 99])) > 0    # the diagonal is not read
    assert _create_rc(linked([0, 4, 1, 0])) == G.GMG_EINVAL     # id >= D*D
    assert _create_rc(linked([0, -1, 1, 0])) == G.GMG_EINVAL
    # sim_opts_t: transfer_mode and gmg_staging take reserved words; the struct size is unchanged
    assert C.sizeof(G._Opts) == 40 and G._Opts.transfer_mode.offset == 24
    assert G._Opts.gmg_staging.offset == 28 and G._Opts.reserved.offset == 32
    hdr = open(os.path.join(ROOT, "include", "gmgsim.h")).read()
    assert re.search(r"int32_t transfer_mode;.*\n\s*int32_t gmg_staging;.*\n\s*int32_t reserved\[2\];", hdr)
    for name, v in (("DEFAULT", 0), ("SHARED", 1), ("L1", 2)):
        assert re.search(r"#define GMG_STAGING_%s %d\b" % (name, v), hdr)
        assert getattr(G, "GMG_STAGING_" + name) == v
    assert "const int32_t* link_id;" in hdr and G._Desc.link_id.offset == C.sizeof(G._Desc) - 8


def test_product_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2608_15762_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".h", ".cpp")):
                src = open(os.path.join(dirpath, f)).read()
                assert not re.search(r"^\s*(from|import)\s+oracle|liboracle|sim_ref", src, re.M), f


def test_nvtx_ranges_are_opt_in_and_balanced(monkeypatch):
    torch = pytest.importorskip("torch")
    calls = []
    monkeypatch.setattr(torch.cuda.nvtx, "range_push", lambda n: calls.append(("push", n)))
    monkeypatch.setattr(torch.cuda.nvtx, "range_pop", lambda: calls.append(("pop",)))

    @G._traced("probe")
    def probe(fail):
        if fail:
            raise ValueError("x")
        return 7
    monkeypatch.setattr(G, "NVTX", False)
    assert probe(False) == 7 and calls == []
    monkeypatch.setattr(G, "NVTX", True)
    assert probe(False) == 7
    with pytest.raises(ValueError):
        probe(True)
    assert calls == [("push", "gmgsim.probe"), ("pop",), ("push", "gmgsim.probe"), ("pop",)]
    assert G.sim_batch.__name__ == "sim_batch" and G.sim_incremental.__wrapped__ is not None
