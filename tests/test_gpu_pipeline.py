"""Calls of several chunks: the library pipelines them over two work
streams and two worklist sets (one chunk's screen and search overlap the
previous chunk's search and top-k).  Results, bounds and the top-k must be
bit-exact with one chunk per call and with the oracle, on every search
path, for ragged chunk sizes."""

import numpy as np
import pytest

import gpu_helpers as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def h(heddle_lib):
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return heddle_lib


@pytest.fixture(scope="module")
def W():
    from paper_2609_34244_gb300 import workloads
    return workloads


def _same(a, b, what):
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (a[key] == b[key]).all(), (what, key)
    for key in ("idx", "T", "nM"):
        assert (a["topk"][key] == b["topk"][key]).all(), (what, key)


@pytest.mark.parametrize("name,n,search", [("stress128", 200003, None), ("dense80", 60011, None),
                                           ("moe48", 50021, None), ("dense80", 30011, "general"),
                                           ("dense32", 40013, "distribute")])
def test_pipelined_chunks_match_one_chunk(h, W, oracle_mod, name, n, search):
    w = W.make_workload(name, seed=3, n=n)
    mode = {None: None, "general": h.SEARCH_GENERAL, "distribute": h.SEARCH_DISTRIBUTE}[search]
    one = G.price_gpu(h, w.cluster, w.model, w.cands, k=32, search=mode, fused=True)
    assert one["errors"] == 0
    for chunk in (65536, 17389):
        for fused in (True, False):
            got = G.price_gpu(h, w.cluster, w.model, w.cands, k=32, search=mode, fused=fused, chunk=chunk,
                              phases=fused)
            assert got["errors"] == 0
            _same(got, one, "%s chunk %d fused %s" % (name, chunk, fused))
            if fused:
                chunks = -(-n // chunk)
                ph = got["phases"]
                assert ph["screen"][1] == chunks and ph["topk"][1] == chunks, ph
                assert ph["search"][0] > 0 and ph["topk"][0] > 0, ph
    # and the oracle on a sample of the pipelined results
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=32, search=mode, fused=True, chunk=17389)
    idx = np.random.default_rng(1).choice(n, 3000, replace=False)
    o = oracle_mod.Oracle(w.cluster, w.model)
    if search == "distribute":
        o.set_split("distribute")
    ref = o.price(G.take(w.cands, idx), threads=8)
    G.assert_same(got, ref, idx=idx, what="%s pipelined sampled" % name)


def test_pipelined_tiling(h, W, oracle_mod):
    w = W.make_workload("moe16", seed=4, n=30011)
    es, ep = w.model["expert_state_bytes"], w.model["expert_param_bytes"]
    one = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, es, ep)
    many = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, es, ep, chunk=4099)
    fused = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, es, ep, chunk=4099, fused=True)
    assert many["errors"] == 0 and fused["errors"] == 0
    for key in ("T", "bottleneck", "n_dp", "status", "bounds", "tiling"):
        assert (one[key] == many[key]).all(), key
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (one[key] == fused[key]).all(), key
    assert one["topk"]["idx"].tolist() == many["topk"]["idx"].tolist() == fused["topk"]["idx"].tolist()


def test_set_chunk_limits(h, W):
    w = W.make_workload("tiny", seed=0)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        for bad in (0, -5, (1 << 20) + 1):
            with pytest.raises(h.HeddleError) as e:
                h.heddle_set_chunk(ctx, bad)
            assert e.value.status == h.E_LIMIT
        h.heddle_set_chunk(ctx, 1)
        h.heddle_set_chunk(ctx, 1 << 20)
    finally:
        h.heddle_destroy(ctx)


def test_tiny_chunks_of_one(h, W, oracle_mod):
    """Chunks of a single candidate: every chunk alternates sets and
    streams."""
    w = W.make_workload("tiny_ext", seed=0)
    ref = oracle_mod.Oracle(w.cluster, w.model).price(w.cands)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, fused=True, chunk=1)
    assert got["errors"] == 0
    G.assert_same(got, ref, what="tiny_ext chunk 1")
    tk = oracle_mod.topk(ref, w.cands["M"], 16)
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()


def _host_price(h, w, batch, experts=None):
    import torch
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        if experts is not None:
            h.heddle_load_experts(ctx, *experts)
        pinned = {k2: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).pin_memory()
                  for k2, v in w.cands.items()}
        n = w.n
        res = {"T": np.zeros(n, np.int64), "bottleneck": np.zeros(n, np.int64), "n_dp": np.zeros(n, np.uint16),
               "status": np.zeros(n, np.uint8), "bounds": np.zeros((33, n), np.uint8)}
        st = h.new_topk_state(16)
        h.heddle_price_topk_host(ctx, pinned, res, st, batch=batch)
        res["topk"] = h.topk_state_to_dict(st)
        res["errors"] = h.heddle_device_errors(ctx)
        return res
    finally:
        h.heddle_destroy(ctx)


def test_host_path_pipelined_batches(h, W):
    """Host buffers in several batches (the last one ragged) on the
    equal-layer path and with expert tiling: the same results and top-k as
    one device call."""
    w = W.make_workload("stress128", seed=5, n=100003)
    dev = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, fused=True)
    got = _host_price(h, w, 16411)
    assert got["errors"] == 0
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (got[key] == dev[key]).all(), key
    assert got["topk"]["idx"].tolist() == dev["topk"]["idx"].tolist()
    wt = W.make_workload("moe16", seed=6, n=20011)
    ex = (wt.model["expert_state_bytes"], wt.model["expert_param_bytes"])
    devt = G.price_tiled_gpu(h, wt.cluster, wt.model, wt.cands, *ex)
    gott = _host_price(h, wt, 3001, experts=ex)
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (gott[key] == devt[key]).all(), key
    assert gott["topk"]["idx"].tolist() == devt["topk"]["idx"].tolist()


def test_host_path_batch_limit(h, W):
    w = W.make_workload("tiny", seed=0)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        with pytest.raises(h.HeddleError) as e:
            h.heddle_price_topk_host(ctx, w.cands, None, h.new_topk_state(4), batch=(1 << 20) + 1)
        assert e.value.status == h.E_LIMIT
    finally:
        h.heddle_destroy(ctx)


def test_threshold_restarts_each_call(h, W, oracle_mod):
    """Inside a top-k pricing the equal-layer search hands the top-k only the
    entries that reach a running threshold below the state's k-th key.  The
    threshold restarts with every call: after a reset, a call whose entries
    are all worse than the previous call's k-th still finds its own exact
    top-k, and calls continuing a full state (two halves) merge exactly,
    through device buffers and through host buffers."""
    import torch
    w = W.make_workload("stress128", seed=7, n=120011)
    ref = oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=8)
    nM = ref["n_dp"].astype(np.int64) * w.cands["M"].astype(np.int64)
    ok = np.nonzero(ref["status"] == 0)[0]
    key = nM[ok].astype(np.float64) / ref["T"][ok].astype(np.float64)
    best = ok[np.argsort(-key, kind="stable")[:3000]]
    worse = {k2: v.copy() for k2, v in w.cands.items()}
    worse["S"][best] = 0  # invalid: every remaining entry is below the first call's k-th
    rest = np.setdiff1d(ok, best)
    expect = [e[0] for e in G.exact_topk(rest, ref["T"][rest], nM[rest], 16)]
    full = [e[0] for e in G.exact_topk(ok, ref["T"][ok], nM[ok], 16)]
    n = w.n
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        h.heddle_set_chunk(ctx, 16411)
        res = h.alloc_results(n, bounds=False)
        state = h.alloc_topk_state()
        for cands, want in ((w.cands, full), (worse, expect)):
            dc = h.cands_to_device(cands)
            h.heddle_topk_reset(ctx, state, 16)
            h.heddle_price_topk(ctx, h.make_candidates(dc), h.make_results(res), state)
            torch.cuda.synchronize()
            assert h.read_topk_state(state)["idx"].tolist() == want
        # two calls on halves of the worse set continue one state
        h.heddle_topk_reset(ctx, state, 16)
        for lo, hi in ((0, n // 2), (n // 2, n)):
            h.heddle_price_topk(ctx, h.make_candidates(dc, lo, hi), h.make_results(res, lo, hi), state)
        torch.cuda.synchronize()
        assert h.read_topk_state(state)["idx"].tolist() == expect
        # host buffers: the same sequence
        for cands, want in ((w.cands, full), (worse, expect)):
            pinned = {k2: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).pin_memory()
                      for k2, v in cands.items()}
            st = h.new_topk_state(16)
            h.heddle_price_topk_host(ctx, pinned, None, st, batch=16411)
            assert h.topk_state_to_dict(st)["idx"].tolist() == want
        assert h.heddle_device_errors(ctx) == 0
    finally:
        h.heddle_destroy(ctx)
