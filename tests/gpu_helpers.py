"""Helpers for the GPU tests: run the CUDA path through the C ABI and the
oracle on the same seeded inputs."""

from __future__ import annotations

import functools

import numpy as np


def price_gpu(h, w_cluster, w_model, cands, k=16, bounds=True, batch=None, count=False, search=None,
              fused=False, phases=False, chunk=None, thread_min=None):
    """Price on the GPU through the C ABI; returns numpy results, the top-k
    and (optionally) the work counters.  ``batch`` splits the candidates into
    consecutive launches merged into one top-k state; ``fused`` prices and
    merges in one call (heddle_price_topk); ``phases`` times the pricing
    phases with the library's events and returns them under "phases";
    ``chunk`` sets the library's chunk size (calls of several chunks are
    pipelined over its work streams); ``thread_min`` sets the general
    search's routing threshold (0: thread kernel whenever it has entries,
    2**31 - 1: warp kernel only)."""
    import torch
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w_cluster)
        h.heddle_load_model(ctx, w_model)
        if search is not None:
            h.heddle_set_search(ctx, search)
        if chunk is not None:
            h.heddle_set_chunk(ctx, chunk)
        if thread_min is not None:
            h.heddle_set_thread_search_min(ctx, thread_min)
        n = int(cands["S"].shape[0])
        dc = h.cands_to_device(cands)
        res = h.alloc_results(n, bounds=False)
        state = h.alloc_topk_state()
        h.heddle_topk_reset(ctx, state, k)
        batch = n if batch is None else batch
        out_bounds = np.zeros((33, n), np.uint8) if bounds else None
        if count:
            h.heddle_count_next(ctx, True)
        if phases:
            h.heddle_time_phases(ctx, True)
        for lo in range(0, max(n, 1), max(batch, 1)):
            hi = min(n, lo + batch)
            if hi <= lo:
                break
            bb = torch.empty((33, hi - lo), dtype=torch.uint8, device="cuda") if bounds else None
            c = h.make_candidates(dc, lo, hi)
            r = h.heddle_results(res["T"].data_ptr() + 8 * lo, res["bottleneck"].data_ptr() + 8 * lo,
                                 res["n_dp"].data_ptr() + 2 * lo, res["status"].data_ptr() + lo,
                                 None if bb is None else bb.data_ptr())
            if fused:
                h.heddle_price_topk(ctx, c, r, state)
            else:
                h.heddle_price_candidates(ctx, c, r)
                h.heddle_topk(ctx, c, r, state)
            if bounds:
                out_bounds[:, lo:hi] = bb.cpu().numpy()
        torch.cuda.synchronize()
        out = h.results_to_numpy(res)
        out["bounds"] = out_bounds
        out["topk"] = h.read_topk_state(state)
        out["errors"] = h.heddle_device_errors(ctx)
        out["search"] = h.heddle_get_search(ctx)
        if count:
            out["counters"] = h.heddle_work_counters(ctx)
        if phases:
            out["phases"] = h.heddle_phase_times(ctx)
        return out
    finally:
        h.heddle_destroy(ctx)


def assert_same(gpu, orc, idx=None, what=""):
    """Bit-exact comparison of every per-candidate field (optionally on the
    sampled indices ``idx``; the oracle then holds results for idx only)."""
    for key in ("status", "n_dp", "T", "bottleneck"):
        g = gpu[key] if idx is None else gpu[key][idx]
        o = orc[key]
        bad = np.nonzero(g != o)[0]
        assert bad.size == 0, "%s %s differs at %d candidates, first %s: gpu %s oracle %s" % (
            what, key, bad.size, bad[:5], g[bad[:5]], o[bad[:5]])
    if gpu.get("bounds") is not None and orc.get("bounds") is not None:
        g = gpu["bounds"] if idx is None else gpu["bounds"][:, idx]
        bad = np.nonzero((g != orc["bounds"]).any(axis=0))[0]
        assert bad.size == 0, "%s bounds differ at %d candidates, first %s" % (what, bad.size, bad[:5])


def exact_topk(idx_all, T, nM, k):
    """Exact top-k of (idx, T, nM) triples by nM/T then smaller idx, using a
    float64 pre-filter and integer cross-multiplication to finish."""
    if len(idx_all) == 0:
        return []
    key = nM.astype(np.float64) / T.astype(np.float64)
    m = min(len(key), max(4 * k, 1000))
    thresh = np.partition(key, len(key) - m)[len(key) - m]
    sel = np.nonzero(key >= thresh)[0]
    items = [(int(idx_all[i]), int(T[i]), int(nM[i])) for i in sel]

    def cmp(a, b):
        l, r = a[2] * b[1], b[2] * a[1]
        if l != r:
            return -1 if l > r else 1
        return -1 if a[0] < b[0] else (1 if a[0] > b[0] else 0)

    items.sort(key=functools.cmp_to_key(cmp))
    return items[:k]


def price_mbs_gpu(h, w_cluster, w_model, cands, levels, profiles=None, bounds=True, search=None, batch=None):
    """Micro-batch-size fill on the GPU through the C ABI (one call, or one
    per ``batch`` candidates); numpy results plus the chosen level ``mbs``."""
    import torch
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w_cluster)
        h.heddle_load_model(ctx, w_model)
        if search is not None:
            h.heddle_set_search(ctx, search)
        h.heddle_load_mbs(ctx, levels, profiles)
        n = int(cands["S"].shape[0])
        dc = h.cands_to_device(cands)
        res = h.alloc_results(n, bounds=bounds)
        mbs = torch.full((max(n, 1),), 255, dtype=torch.uint8, device="cuda")
        if batch is None:
            h.heddle_price_mbs(ctx, h.make_candidates(dc), h.make_results(res), mbs)
        else:
            for lo in range(0, n, batch):
                hi = min(n, lo + batch)
                h.heddle_price_mbs(ctx, h.make_candidates(dc, lo, hi), h.make_results(res, lo, hi), mbs[lo:hi])
        torch.cuda.synchronize()
        out = h.results_to_numpy(res)
        out["mbs"] = mbs[:n].cpu().numpy()
        out["errors"] = h.heddle_device_errors(ctx)
        return out
    finally:
        h.heddle_destroy(ctx)


def take(cands, idx):
    """The candidates at indices ``idx`` (a host SoA copy)."""
    return {"S": cands["S"][idx].copy(), "M": cands["M"][idx].copy(),
            "code": np.ascontiguousarray(cands["code"][:, idx])}


def price_tiled_gpu(h, w_cluster, w_model, cands, expert_state, expert_param, k=16, fused=False, batch=None,
                    chunk=None):
    """Expert tiling on the GPU through the C ABI: heddle_price_tiled (with
    the tiling planes) and heddle_topk, or heddle_price_topk with ``fused``;
    ``batch`` splits the candidates into consecutive calls."""
    import torch
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w_cluster)
        h.heddle_load_model(ctx, w_model)
        h.heddle_load_experts(ctx, expert_state, expert_param)
        if chunk is not None:
            h.heddle_set_chunk(ctx, chunk)
        n = int(cands["S"].shape[0])
        dc = h.cands_to_device(cands)
        res = h.alloc_results(n, bounds=False)
        state = h.alloc_topk_state()
        h.heddle_topk_reset(ctx, state, k)
        batch = n if batch is None else batch
        out_bounds = np.zeros((33, n), np.uint8)
        out_tiling = np.zeros((32, n), np.uint8)
        for lo in range(0, n, max(batch, 1)):
            hi = min(n, lo + batch)
            bb = torch.empty((33, hi - lo), dtype=torch.uint8, device="cuda")
            tt = torch.full((32, hi - lo), 0xEE, dtype=torch.uint8, device="cuda")
            c = h.make_candidates(dc, lo, hi)
            r = h.heddle_results(res["T"].data_ptr() + 8 * lo, res["bottleneck"].data_ptr() + 8 * lo,
                                 res["n_dp"].data_ptr() + 2 * lo, res["status"].data_ptr() + lo, bb.data_ptr())
            if fused:
                h.heddle_price_topk(ctx, c, r, state)
            else:
                h.heddle_price_tiled(ctx, c, r, tt)
                h.heddle_topk(ctx, c, r, state)
            out_bounds[:, lo:hi] = bb.cpu().numpy()
            out_tiling[:, lo:hi] = tt.cpu().numpy()
        torch.cuda.synchronize()
        out = h.results_to_numpy(res)
        out["bounds"] = out_bounds
        out["tiling"] = None if fused else out_tiling
        out["topk"] = h.read_topk_state(state)
        out["errors"] = h.heddle_device_errors(ctx)
        out["search"] = h.heddle_get_search(ctx)
        return out
    finally:
        h.heddle_destroy(ctx)
