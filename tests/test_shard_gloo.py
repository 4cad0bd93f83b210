"""Multi-rank sharding of one batch, on CPU with world-size-2 gloo groups.

Each rank takes its contiguous slot range and its export budget with the
benchmark's own functions (``bench.shard_queries``, ``bench.shard_budget``:
an all-gather of every rank's undischarged count), checks its range (here
with the CPU oracle: no GPU takes part), and rank 0 merges verdict counts and
exports.  The merged result must equal the single-rank result byte for
byte.
"""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2609_19611_gb300 import shard
from paper_2609_19611_gb300 import workloads as W


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _case():
    return W.config(2, N=2, Ci=2, H=8, W=8, Co=3)


def _check(ref, cand, locs, budget):
    R, C = oracle.Program(ref), oracle.Program(cand)
    kr, kc = R.keys(locs, nthreads=1), C.keys(locs, nthreads=1)
    cones = (R.cone_runs(locs, 1), C.cone_runs(locs, 1))
    v, f, blob, need = oracle.compare(R, C, locs, kr, kc, cones=cones, budget=budget)
    stats = {"n_discharged": int((v == 0).sum()), "n_exported": int((v == 1).sum()),
             "n_unexported": int((v == 2).sum()),
             "n_cone_differs": int(((f & 1) != 0).sum()), "n_bot_ref": int(((f & 2) != 0).sum()),
             "n_bot_cand": int(((f & 4) != 0).sum())}
    return v, f, blob, stats


def _rank(rank, world, port, budget, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ref, cand = _case()
        locs = W.make_queries(2, 2 * 8 * 8, n=300, seed=11)
        # the benchmark's own host logic: its slot range, then (from every
        # rank's undischarged count, one all-gather) its export budget
        import bench
        mine, lo = bench.shard_queries(locs, world, rank)
        R, C = oracle.Program(ref), oracle.Program(cand)
        und = int((~(R.keys(mine, nthreads=1) == C.keys(mine, nthreads=1)).all(axis=1)).sum())
        b = bench.shard_budget(und, budget, world, rank)
        v, f, blob, stats = _check(ref, cand, mine, b)
        gathered = [None] * world
        dist.all_gather_object(gathered, (lo, v.tolist(), f.tolist(), blob, stats))
        if rank == 0:
            q.put(gathered)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("budget", [0, 5, 40, 1000])
def test_two_rank_shards_merge_to_single_rank_result(budget):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, budget, q)) for r in range(2)]
    for p in procs:
        p.start()
    gathered = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    ref, cand = _case()
    locs = W.make_queries(2, 2 * 8 * 8, n=300, seed=11)
    v1, f1, blob1, stats1 = _check(ref, cand, locs, budget)
    offs = [g[0] for g in gathered]
    v = np.concatenate([np.asarray(g[1], dtype=np.uint8) for g in gathered])
    f = np.concatenate([np.asarray(g[2], dtype=np.uint8) for g in gathered])
    assert np.array_equal(v, v1) and np.array_equal(f, f1)
    assert shard.merge_stats([g[4] for g in gathered]) == stats1
    merged = shard.merge_exports([g[3] for g in gathered], offs)
    assert merged == blob1


def test_shard_ranges_cover_the_batch():
    for n in (0, 1, 7, 300):
        for world in (1, 2, 3, 8):
            rs = [shard.shard_range(n, world, r) for r in range(world)]
            assert rs[0][0] == 0 and rs[-1][1] == n
            assert all(a[1] == b[0] for a, b in zip(rs, rs[1:]))
            assert max(h - l for l, h in rs) - min(h - l for l, h in rs) <= 1


def test_rank_budgets():
    assert shard.rank_budgets([3, 4, 5], 6) == [3, 3, 0]
    assert shard.rank_budgets([0, 4], 2) == [0, 2]
    assert shard.rank_budgets([3, 4], 0) == [0, 0]
