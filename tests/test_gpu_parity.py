"""CUDA path (through the C ABI) against the CPU oracle: bit-exact partitions,
iteration times, DP degrees, statuses and top-k on seeded inputs."""

import json
import os

import numpy as np
import pytest

import gpu_helpers as G
import pin_checks as PC

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


# sizes span many CTAs (128 threads each) and end on a ragged tail
SMALL = [("tiny", None), ("tiny_ext", None), ("dense32", 6007), ("dense80", 1531),
         ("moe48", 6011), ("moe16", 4001), ("stress128", 613)]


# the equal-layer search runs on models whose layers all cost the same
EQUAL = {"dense32", "dense80", "stress128"}


# the general search's two routes forced: the thread-per-entry kernel
# wherever it has entries, or the warp-per-entry kernel for every entry
ROUTES = {"auto": (0, None), "general": (1, None), "thread": (1, 0), "warp": (1, 2**31 - 1)}


@pytest.mark.parametrize("name,n", SMALL)
@pytest.mark.parametrize("seed", [0, 1])
@pytest.mark.parametrize("route", list(ROUTES))
def test_parity_small(h, W, oracle_mod, name, n, seed, route):
    search, thread_min = ROUTES[route]
    w = W.make_workload(name, seed=seed, n=n)
    orc = oracle_mod.Oracle(w.cluster, w.model)
    ref = orc.price(w.cands, threads=8)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, search=search, thread_min=thread_min)
    assert got["errors"] == 0
    assert got["search"] == (2 if (search == 0 and name in EQUAL) else 1)
    G.assert_same(got, ref, what=name)
    tk = oracle_mod.topk(ref, w.cands["M"], 16)
    assert got["topk"]["count"] == tk["count"]
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()
    assert got["topk"]["T"].tolist() == tk["T"].tolist()
    assert got["topk"]["nM"].tolist() == tk["nM"].tolist()


def test_thread_search_defers_to_warp_search(h, W, oracle_mod):
    """moe16 through the thread-per-entry search: entries whose bracket
    falls below the single-fit threshold are handed to the warp search
    (counted twice: the interval-test counters see both kernels), and the
    results still equal the oracle's."""
    w = W.make_workload("moe16", seed=0, n=4001)
    ref = oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=8)
    both = G.price_gpu(h, w.cluster, w.model, w.cands, search=1, thread_min=0, count=True)
    warp = G.price_gpu(h, w.cluster, w.model, w.cands, search=1, thread_min=2**31 - 1, count=True)
    for got in (both, warp):
        assert got["errors"] == 0
        G.assert_same(got, ref, what="moe16")
    assert both["counters"]["priced"] > warp["counters"]["priced"], "no entry was handed on"


@pytest.mark.parametrize("name", ["tiny", "dense32", "dense80", "moe48", "stress128"])
def test_tables_match_oracle(h, W, oracle_mod, name):
    w = W.make_workload(name, n=10)
    tab = oracle_mod.Oracle(w.cluster, w.model).tables()
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        q, p2p = h.heddle_get_tables(ctx, len(w.cluster["tflops"]), len(w.model["flops"]))
    finally:
        h.heddle_destroy(ctx)
    assert (q == tab["q"]).all()
    assert (p2p == tab["p2p"]).all()


def test_hand_golden_on_gpu(h, oracle_mod):
    """The GPU reproduces the hand-worked end-to-end prices directly."""
    with open(os.path.join(PC.GOLDEN, "hand_pricing.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        orc, cands, L = PC.oracle_for(oracle_mod, case)
        W = PC._workloads()
        cl = case["cluster"]
        cluster = W.make_cluster(cl["tflops"], cl["mem_bytes"], cl["intra_bw"], [tuple(x) for x in cl["nodes"]])
        m = case["model"]
        model = W.make_model(m["flops"], m["param_bytes"], m["state_bytes"], m["act_bytes"], m["ar_bytes"],
                             m["a2a_bytes"], m["boundary_bytes"], moe=m["moe"])
        got = G.price_gpu(h, cluster, model, cands, k=len(case["expect"]))
        for c, exp in enumerate(case["expect"]):
            assert int(got["status"][c]) == exp["status"], case["name"]
            assert int(got["n_dp"][c]) == exp["n_dp"], case["name"]
            assert int(got["T"][c]) == exp["T"], case["name"]
            assert int(got["bottleneck"][c]) == exp["bottleneck"], case["name"]
            if exp["bounds"] is not None:
                S = int(cands["S"][c])
                assert got["bounds"][: S + 1, c].tolist() == exp["bounds"], case["name"]
        if "topk_order" in case:
            assert got["topk"]["idx"].tolist() == case["topk_order"], case["name"]


def test_raw_partitions_on_gpu(h, W, oracle_mod):
    """Random small instances where memory binds often: GPU vs oracle DP
    (which is itself checked against brute force)."""
    rng = np.random.default_rng(5)
    for trial in range(30):
        L = int(rng.integers(1, 24))
        nt = int(rng.integers(1, 4))
        cluster = W.make_cluster(rng.uniform(100, 1000, nt), rng.integers(1, 6, nt) * 10**9,
                                 rng.integers(1, 10, nt) * 10**11,
                                 [(g % nt, int(rng.choice([1, 2, 4, 8])), int(rng.integers(1, 50)) * 10**9)
                                  for g in range(nt + int(rng.integers(0, 4)))])
        model = W.make_model(rng.uniform(0, 5e12, L), rng.integers(0, 10**9, L), rng.integers(0, 4 * 10**9, L),
                             rng.integers(0, 10**9, L), rng.integers(0, 10**8, L), 0,
                             int(rng.integers(0, 10**8)), moe=bool(rng.random() < 0.3))
        n = 500
        S = rng.integers(1, min(L, 32) + 1, n)
        code = np.zeros((32, n), np.uint8)
        code[:] = W.encode(rng.integers(0, nt, (32, n)), rng.integers(0, 4, (32, n)))
        code[np.arange(32)[:, None] >= S[None, :]] = 0
        cands = W.make_cands(S, rng.integers(1, 64, n), code)
        ref = oracle_mod.Oracle(cluster, model).price(cands)
        got = G.price_gpu(h, cluster, model, cands)
        assert got["errors"] == 0
        G.assert_same(got, ref, what="trial %d" % trial)


def test_equal_layer_random_instances(h, W, oracle_mod):
    """Random equal-layer models (one layer repeated, so the closed-form
    search runs), memory often binding, P2P and replication on: GPU in both
    search modes vs the oracle DP."""
    rng = np.random.default_rng(17)
    for trial in range(40):
        L = int(rng.integers(1, 64))
        nt = int(rng.integers(1, 5))
        cluster = W.make_cluster(rng.uniform(50, 1000, nt), rng.integers(1, 12, nt) * 10**9,
                                 rng.integers(1, 10, nt) * 10**11,
                                 [(g % nt, int(rng.choice([1, 2, 3, 4, 8])), int(rng.integers(1, 50)) * 10**9)
                                  for g in range(nt + int(rng.integers(0, 6)))])
        flops = float(rng.uniform(0, 5e12)) if rng.random() < 0.9 else 0.0
        model = W.make_model(np.full(L, flops), int(rng.integers(0, 10**9)), int(rng.integers(0, 2 * 10**9)),
                             int(rng.integers(0, 10**9)), int(rng.integers(0, 10**8)), 0,
                             int(rng.integers(0, 10**8)), moe=bool(rng.random() < 0.3))
        n = 700
        S = rng.integers(1, min(L, 32) + 1, n)
        code = W.encode(rng.integers(0, nt, (32, n)), rng.integers(0, 4, (32, n)))
        code[np.arange(32)[:, None] >= S[None, :]] = 0
        cands = W.make_cands(S, rng.integers(1, 300, n), code)
        ref = oracle_mod.Oracle(cluster, model).price(cands)
        for search in (0, 1):
            got = G.price_gpu(h, cluster, model, cands, search=search)
            assert got["errors"] == 0
            assert got["search"] == (2 if search == 0 else 1)
            G.assert_same(got, ref, what="trial %d search %d" % (trial, search))


def test_batching_and_launch_shape_do_not_change_results(h, W, oracle_mod):
    w = W.make_workload("moe48", seed=0, n=5000)
    a = G.price_gpu(h, w.cluster, w.model, w.cands, k=64)
    assert (a["status"] == 0).sum() > 20  # the search really runs
    b = G.price_gpu(h, w.cluster, w.model, w.cands, k=64, batch=777)
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (a[key] == b[key]).all(), key
    for key in ("idx", "T", "nM"):
        assert (a["topk"][key] == b["topk"][key]).all()
    c = G.price_gpu(h, w.cluster, w.model, w.cands, k=64, count=True)
    for key in ("T", "bottleneck", "n_dp", "status"):
        assert (a[key] == c[key]).all(), key
    assert c["counters"]["checks"] > 0 and c["counters"]["priced"] > 0
    # phase timing: same results, one screen and one search launch per
    # chunk, one top-k launch per fused chunk
    chunks = -(-5000 // 777)
    for fused in (False, True):
        d = G.price_gpu(h, w.cluster, w.model, w.cands, k=64, batch=777, fused=fused, phases=True)
        for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
            assert (b[key] == d[key]).all(), key
        assert d["topk"]["idx"].tolist() == b["topk"]["idx"].tolist()
        ph = d["phases"]
        assert ph["screen"][1] == chunks and ph["search"][1] == chunks, ph
        assert ph["screen"][0] > 0 and ph["search"][0] > 0, ph
        if fused:
            assert ph["topk"][1] == chunks and ph["topk"][0] > 0, ph
        else:
            assert ph["topk"] == (0.0, 0), ph


@pytest.mark.parametrize("name,n,seed", [("dense32", 20011, 0), ("moe48", 20011, 0), ("tiny_ext", None, 0),
                                         ("stress128", 30011, 1), ("dense80", 9001, 2)])
@pytest.mark.parametrize("k", [1, 16, 64])
def test_fused_price_topk(h, W, oracle_mod, name, n, seed, k):
    """heddle_price_topk (top-k fused into the search) == price then topk ==
    the oracle's top-k, for several k, batch splits and both searches."""
    w = W.make_workload(name, seed=seed, n=n)
    ref = oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=8)
    tk = oracle_mod.topk(ref, w.cands["M"], k)
    for search in (0, 1):
        for batch in (None, 7001):
            got = G.price_gpu(h, w.cluster, w.model, w.cands, k=k, bounds=False, batch=batch, search=search,
                              fused=True)
            assert got["errors"] == 0
            G.assert_same(got, ref, what="%s fused" % name)
            assert got["topk"]["idx"].tolist() == tk["idx"].tolist(), (name, k, search, batch)
            assert got["topk"]["T"].tolist() == tk["T"].tolist()
            assert got["topk"]["nM"].tolist() == tk["nM"].tolist()


def test_edge_cases(h, W, oracle_mod):
    # n = 0 is a no-op; n = 1
    w = W.make_workload("dense32", n=1)
    got = G.price_gpu(h, w.cluster, w.model, w.cands)
    G.assert_same(got, oracle_mod.Oracle(w.cluster, w.model).price(w.cands))
    empty = W.make_cands(np.zeros(0, np.uint8), np.zeros(0, np.uint16), np.zeros((8, 0), np.uint8))
    got = G.price_gpu(h, w.cluster, w.model, empty)
    assert got["topk"]["count"] == 0
    # maximum sizes: 255 layers, 32 stages, 8 types, k = 64
    rng = np.random.default_rng(11)
    L = 255
    cluster = W.make_cluster(rng.uniform(50, 1000, 8), rng.integers(100, 400, 8) * 10**9,
                             rng.integers(1, 10, 8) * 10**11,
                             [(g, int(s), 25 * 10**9) for g in range(8) for s in (8, 8, 4, 2)])
    model = W.make_model(rng.uniform(1e11, 1e12, L), 10**8, 8 * 10**8, 10**7, 10**7, 0, 10**7)
    n = 3001
    S = np.full(n, 32, np.uint8)
    S[::7] = rng.integers(1, 32, S[::7].shape[0])
    code = W.encode(rng.integers(0, 8, (32, n)), rng.integers(0, 4, (32, n)))
    code[np.arange(32)[:, None] >= S[None, :]] = 0
    cands = W.make_cands(S, rng.integers(1, 65536, n), code)
    ref = oracle_mod.Oracle(cluster, model).price(cands, threads=8)
    got = G.price_gpu(h, cluster, model, cands, k=64)
    G.assert_same(got, ref, what="max sizes")
    tk = oracle_mod.topk(ref, cands["M"], 64)
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()
    # degenerate: zero-cost layers, every candidate S = 1, all invalid
    model0 = W.make_model(np.zeros(L), 0, 0, 0, 0, 0, 0)
    ref = oracle_mod.Oracle(cluster, model0).price(cands, threads=8)
    got = G.price_gpu(h, cluster, model0, cands, k=64)
    G.assert_same(got, ref, what="zero costs")
    bad = W.make_cands(S, np.zeros(n, np.uint16), code)
    got = G.price_gpu(h, cluster, model, bad)
    assert (got["status"] == 3).all() and got["topk"]["count"] == 0


def test_host_buffer_path_matches_device_path(h, W):
    import torch
    w = W.make_workload("dense80", seed=2, n=20011)
    dev = G.price_gpu(h, w.cluster, w.model, w.cands, k=16)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        pinned = {k2: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).pin_memory()
                  for k2, v in w.cands.items()}
        n = w.n
        res = {"T": np.zeros(n, np.int64), "bottleneck": np.zeros(n, np.int64), "n_dp": np.zeros(n, np.uint16),
               "status": np.zeros(n, np.uint8), "bounds": np.zeros((33, n), np.uint8)}
        st = h.new_topk_state(16)
        h.heddle_price_topk_host(ctx, pinned, res, st, batch=6000)
        tk = h.topk_state_to_dict(st)
    finally:
        h.heddle_destroy(ctx)
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (res[key] == dev[key]).all(), key
    assert tk["idx"].tolist() == dev["topk"]["idx"].tolist()


def test_call_errors(h, W):
    w = W.make_workload("dense32", n=10)
    ctx = h.heddle_create(0)
    try:
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(w.n)
        with pytest.raises(h.HeddleError) as e:
            h.heddle_price_candidates(ctx, dc, res)
        assert e.value.status == 2  # no cluster / model
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        c = h.make_candidates(dc)
        c.s_max = 0
        with pytest.raises(h.HeddleError) as e:
            h.heddle_price_candidates(ctx, c, res)
        assert e.value.status == 1
        bad = dict(w.cluster)
        bad["node_gpus"] = np.zeros_like(bad["node_gpus"])
        with pytest.raises(h.HeddleError):
            h.heddle_load_cluster(ctx, bad)
        with pytest.raises(h.HeddleError) as e:
            h.heddle_topk_reset(ctx, h.alloc_topk_state(), 65)
        assert e.value.status == 3
        # the routing setting: a NULL context is refused; any value is taken
        assert h.load_library().heddle_set_thread_search_min(None, 0) == 1
        for v in (-5, 0, 2**31 - 1):
            h.heddle_set_thread_search_min(ctx, v)
    finally:
        h.heddle_destroy(ctx)
