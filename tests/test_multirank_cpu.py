"""The multi-rank path on CPU with gloo (world size 2).  Every rank takes a
contiguous block of each half of the candidates -- full placements and
incremental move lists against a replicated base -- with uneven block sizes
and no data-path exchange; the per-rank bests are combined by one small
all_gather into the best over all candidates, with global indices that list
the full placements first.  The per-rank evaluation here is the oracle (no
GPU); the test covers the partition, the index mapping and the cross-rank
selection."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
N_FULL, N_INC = 37, 23          # uneven over two ranks
CAP = 728_735_855               # a tight capacity: some candidates are infeasible


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _workload():
    import sys
    sys.path.insert(0, ROOT)
    from paper_2608_15762_gb300 import workloads as W
    wl = W.config1()
    wl.desc.cap[:] = CAP
    base = wl.full_rows([0])[0, :wl.desc.n_ops].copy()
    moves = W.random_moves(3, N_INC, base, wl.desc.n_dev, max_moves=6)
    return wl, base, moves


def _rank_main(rank, world, port, q):
    import sys
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    from oracle import oracle as O
    from paper_2608_15762_gb300 import gmgsim as G
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl, base, moves = _workload()
    fk = G.shard_block(rank, world, N_FULL)
    ik = G.shard_block(rank, world, N_INC)
    sf, _, _ = O.simulate_batch(wl.desc, wl.full_rows(fk), nthreads=1)
    si, _, _ = O.incremental_batch(wl.desc, base, moves.subset(ik), nthreads=1)
    s = np.concatenate([sf, si])
    k, sc = O.select_best(s, 0)
    best = torch.tensor([k, sc], dtype=torch.int64)
    res = G.select_best_across_ranks(best, G.two_half_index(len(fk), fk.start, N_FULL, ik.start))
    q.put((rank, list(fk), list(ik), res, int(s.shape[0])))
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_partitioned_halves_and_global_best(world):
    from oracle import oracle as O
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = [q.get(timeout=180) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    got.sort()
    # each candidate of each half is simulated by exactly one rank
    full = [set(g[1]) for g in got]
    inc = [set(g[2]) for g in got]
    assert not (full[0] & full[1]) and full[0] | full[1] == set(range(N_FULL))
    assert not (inc[0] & inc[1]) and inc[0] | inc[1] == set(range(N_INC))
    assert sum(g[4] for g in got) == N_FULL + N_INC
    assert {len(f) for f in full} == {18, 19}
    wl, base, moves = _workload()
    sf, _, _ = O.simulate_batch(wl.desc, wl.full_rows(range(N_FULL)), nthreads=2)
    si, _, _ = O.incremental_batch(wl.desc, base, moves, nthreads=2)
    s = np.concatenate([sf, si])
    want = O.select_best(s, 0)
    assert 0 < (s["viol_flag"] == 1).sum() < len(s)
    for _, _, _, res, _ in got:
        assert tuple(res) == want


def test_winner_in_the_incremental_half_maps_past_every_full_placement():
    """A rank's local index beyond its full block maps into the incremental
    half, after all full placements of every rank."""
    from paper_2608_15762_gb300 import gmgsim as G
    f = G.two_half_index(18, 19, 37, 11)
    assert [f(0), f(17), f(18), f(29)] == [19, 36, 48, 59]
    assert [len(G.shard_block(r, 3, 10)) for r in range(3)] == [3, 3, 4]
    assert G.shard_block(2, 3, 10) == range(6, 10)
