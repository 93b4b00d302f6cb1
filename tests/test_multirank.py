"""Sharded pricing across ranks (world size 2, gloo, CPU): each rank prices
its shard with the oracle and the host-side merge of the per-rank top-k lists
equals the top-k of the whole set."""

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


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    from oracle import oracle as O
    from paper_2609_34244_gb300 import shard, workloads as W
    g = shard.init(world)
    w = W.make_workload("moe48", seed=4, n=3001)
    lo, hi = shard.shard_range(w.n, rank, world)
    sub = W.slice_cands(w.cands, lo, hi)
    r = O.Oracle(w.cluster, w.model).price(sub)
    local = O.topk(r, sub["M"], 16, base_index=lo)
    merged = shard.merge_topk_across_ranks(g, local, 16)
    t = shard.max_over_ranks(g, float(rank))
    shard.barrier(g)
    out[rank] = (merged["idx"].tolist(), t)
    import torch.distributed as dist
    dist.destroy_process_group()


def test_two_rank_merge_equals_unsharded(oracle_mod):
    from paper_2609_34244_gb300 import workloads as W
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    w = W.make_workload("moe48", seed=4, n=3001)
    full = oracle_mod.topk(oracle_mod.Oracle(w.cluster, w.model).price(w.cands), w.cands["M"], 16)
    assert out[0][0] == full["idx"].tolist() == out[1][0]
    assert out[0][1] == 1.0 and out[1][1] == 1.0


def test_shard_ranges_cover_exactly():
    from paper_2609_34244_gb300 import shard
    for n in (0, 1, 7, 1000):
        for world in (1, 2, 3, 8):
            rs = [shard.shard_range(n, r, world) for r in range(world)]
            assert rs[0][0] == 0 and rs[-1][1] == n
            assert all(rs[i][1] == rs[i + 1][0] for i in range(world - 1))


def _gpu_worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch
    from paper_2609_34244_gb300 import _build, shard, workloads as W
    _build.build()
    from paper_2609_34244_gb300 import heddle as h
    torch.cuda.set_device(0)
    g = shard.init(world)
    w = W.make_workload("dense32", seed=5, n=200_003)
    lo, hi = shard.shard_range(w.n, rank, world)
    sub = W.slice_cands(w.cands, lo, hi)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        h.heddle_set_chunk(ctx, 65_536)
        dc = h.cands_to_device(sub)
        res = h.alloc_results(hi - lo)
        state = h.alloc_topk_state()
        h.heddle_topk_reset(ctx, state, 16)
        h.heddle_price_topk(ctx, h.make_candidates(dc, base_index=lo), h.make_results(res), state)
        torch.cuda.synchronize()
        local = h.read_topk_state(state)
        errors = h.heddle_device_errors(ctx)
    finally:
        h.heddle_destroy(ctx)
    merged = shard.merge_topk_across_ranks(g, local, 16)
    shard.barrier(g)
    out[rank] = (merged["idx"].tolist(), merged["T"].tolist(), merged["nM"].tolist(), errors)
    import torch.distributed as dist
    dist.destroy_process_group()


@pytest.mark.gpu
def test_two_rank_library_merge_on_one_gpu(oracle_mod, heddle_lib):
    """Two processes share cuda:0, each prices its shard through libheddle
    (global indices via base_index), and the host-side gloo merge of their
    top-16 lists equals the oracle's top-16 of the whole set.  The ranks'
    kernels never wait on each other; only the host merge exchanges data."""
    from paper_2609_34244_gb300 import workloads as W
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_gpu_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=600)
        assert p.exitcode == 0
    w = W.make_workload("dense32", seed=5, n=200_003)
    full = oracle_mod.topk(oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=8, bounds=False),
                           w.cands["M"], 16)
    for r in range(2):
        idx, T, nM, errors = out[r]
        assert errors == 0
        assert idx == full["idx"].tolist()
        assert T == full["T"].tolist()
        assert nM == full["nM"].tolist()
