"""The multi-rank path on CPU with gloo (world size 2): each rank takes its
own block of candidates (no data-path exchange) and the per-rank bests are
combined by one small all_gather into the best over all candidates.  The
per-rank evaluation here is the oracle (no GPU); the test covers the
sharding and the cross-rank selection."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank_main(rank, world, port, per_rank, q):
    import sys
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    from oracle import oracle as O
    from paper_2608_15762_gb300 import gmgsim as G
    from paper_2608_15762_gb300 import workloads as W
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl = W.config1()
    wl.desc.cap[:] = 728_735_855   # a tight capacity: some candidates are infeasible
    ks = G.shard_range(rank, per_rank)
    s, _, _ = O.simulate_batch(wl.desc, wl.full_rows(ks), nthreads=1)
    k, sc = O.select_best(s, 0)
    best = torch.tensor([k, sc], dtype=torch.int64)
    res = G.select_best_across_ranks(best, ks.start)
    q.put((rank, list(ks), res))
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_sharded_candidates_and_global_best(world):
    from oracle import oracle as O
    from paper_2608_15762_gb300 import workloads as W
    per_rank = 40
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, per_rank, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    got.sort()
    blocks = [set(g[1]) for g in got]
    assert not (blocks[0] & blocks[1]) and len(blocks[0] | blocks[1]) == world * per_rank
    wl = W.config1()
    wl.desc.cap[:] = 728_735_855
    s, _, _ = O.simulate_batch(wl.desc, wl.full_rows(range(world * per_rank)), nthreads=2)
    want = O.select_best(s, 0)
    assert 0 < (s["viol_flag"] == 1).sum() < len(s)
    for _, _, res in got:
        assert tuple(res) == want
