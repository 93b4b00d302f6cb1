"""Expert tiling (§5.3 "Expert tiling") on the GPU through the C ABI
against the oracle on the same seeded inputs: bit-exact T, bottleneck,
n_dp, status, bounds, the chosen tiling of every stage, and the top-k."""

import json
import os

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


def _experts(w):
    return w.model["expert_state_bytes"], w.model["expert_param_bytes"]


def _oracle(oracle_mod, w):
    return oracle_mod.Oracle(w.cluster, w.model).set_experts(*_experts(w))


def _assert_tiling(got, ref, what):
    ok = ref["status"] == 0
    bad = np.nonzero((got["tiling"][:, ok] != ref["tiling"][:, ok]).any(axis=0))[0]
    assert bad.size == 0, "%s tiling differs at %d OK candidates" % (what, bad.size)
    assert (got["tiling"][:, ~ok] == 0).all(), what + " tiling planes of non-OK candidates"


@pytest.mark.parametrize("name,n", [("moe16", 20011), ("moe48", 40009)])
@pytest.mark.parametrize("seed", [0, 1])
def test_tiling_parity(h, W, oracle_mod, name, n, seed):
    w = W.make_workload(name, seed=seed, n=n)
    ref = _oracle(oracle_mod, w).price(w.cands, threads=8, tiling=True)
    got = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, *_experts(w))
    assert got["errors"] == 0
    assert got["search"] == h.SEARCH_TILED
    assert (ref["status"] == 0).sum() > 50, name
    G.assert_same(got, ref, what="%s tiled" % name)
    _assert_tiling(got, ref, name)
    tk = oracle_mod.topk(ref, w.cands["M"], 16)
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()


def test_tiling_batches_and_fused_topk(h, W, oracle_mod):
    """Several calls with a ragged tail, and the fused price + top-k call."""
    w = W.make_workload("moe16", seed=2, n=9973)
    ref = _oracle(oracle_mod, w).price(w.cands, threads=8, tiling=True)
    tk = oracle_mod.topk(ref, w.cands["M"], 16)
    got = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, *_experts(w), batch=4096)
    G.assert_same(got, ref, what="moe16 batched")
    _assert_tiling(got, ref, "moe16 batched")
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()
    fused = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, *_experts(w), fused=True)
    G.assert_same(fused, ref, what="moe16 fused")
    assert fused["topk"]["idx"].tolist() == tk["idx"].tolist()


def test_tiling_hand_cases(h, W):
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_tiling.json")
    for case in json.load(open(path))["cases"]:
        cl = W.make_cluster(case["tflops"], case["mem_bytes"], case["intra_bw"], [tuple(x) for x in case["nodes"]])
        md = W.make_model(case["flops"], case["param_bytes"], case["state_bytes"], case["act_bytes"],
                          case["ar_bytes"], case["a2a_bytes"], case["boundary_bytes"], moe=True)
        cands = W.from_structures([[tuple(s) for s in case["stages"]]], [case["M"]])
        got = G.price_tiled_gpu(h, cl, md, cands, case["expert_state"], case["expert_param"])
        S = len(case["stages"])
        e = case["expect"]
        assert int(got["status"][0]) == e["status"], case["name"]
        assert int(got["T"][0]) == e["T"], case["name"]
        assert int(got["bottleneck"][0]) == e["bottleneck"], case["name"]
        assert got["bounds"][: S + 1, 0].tolist() == e["bounds"], case["name"]
        assert got["tiling"][:S, 0].tolist() == e["tiling"], case["name"]


def test_tiling_without_experts_is_the_plain_price(h, W):
    """Zero expert bytes on a dense model: identical to untiled pricing, and
    every stage keeps EP over all its devices."""
    w = W.make_workload("dense80", seed=4, n=3001)
    L = int(w.model["flops"].shape[0])
    z = np.zeros(L, np.int64)
    plain = G.price_gpu(h, w.cluster, w.model, w.cands)
    tiled = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, z, z)
    G.assert_same(tiled, plain, what="dense80 zero experts")
    ok = plain["status"] == 0
    S = w.cands["S"][ok]
    j = (w.cands["code"][:, ok] >> 3) & 3
    live = np.arange(j.shape[0])[:, None] < S[None, :]
    assert (tiled["tiling"][: j.shape[0], ok][live] == j[live]).all()
    assert plain["topk"]["idx"].tolist() == tiled["topk"]["idx"].tolist()


def test_tiling_call_errors(h, W):
    import torch
    w = W.make_workload("moe16", seed=0, n=64)
    es, ep = _experts(w)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(64, bounds=True)
        with pytest.raises(h.HeddleError) as ei:  # no experts loaded
            h.heddle_price_tiled(ctx, dc, res)
        assert ei.value.status == h.E_STATE
        bad = np.array(es)
        bad[1] = int(w.model["state_bytes"][1]) + 1
        with pytest.raises(h.HeddleError) as ei:  # expert part above the layer's state
            h.heddle_load_experts(ctx, bad, ep)
        assert ei.value.status == h.E_ARG
        with pytest.raises(h.HeddleError) as ei:  # wrong layer count
            h.heddle_load_experts(ctx, es[:-1], ep[:-1])
        assert ei.value.status == h.E_ARG
        h.heddle_load_experts(ctx, es, ep)
        assert h.heddle_get_search(ctx) == h.SEARCH_TILED
        h.heddle_set_search(ctx, h.SEARCH_DISTRIBUTE)
        with pytest.raises(h.HeddleError) as ei:  # tiling prices the min-max split only
            h.heddle_price_candidates(ctx, dc, res)
        assert ei.value.status == h.E_STATE
        h.heddle_set_search(ctx, h.SEARCH_AUTO)
        h.heddle_load_mbs(ctx, 2)
        with pytest.raises(h.HeddleError) as ei:
            h.heddle_price_mbs(ctx, dc, res)
        assert ei.value.status == h.E_STATE
        h.heddle_price_tiled(ctx, dc, res)
        torch.cuda.synchronize()
        # loading a model turns tiling off
        h.heddle_load_model(ctx, w.model)
        assert h.heddle_get_search(ctx) != h.SEARCH_TILED
        with pytest.raises(h.HeddleError) as ei:
            h.heddle_price_tiled(ctx, dc, res)
        assert ei.value.status == h.E_STATE
        # both NULL turn it off explicitly
        h.heddle_load_experts(ctx, es, ep)
        h.heddle_load_experts(ctx, None, None)
        assert h.heddle_get_search(ctx) != h.SEARCH_TILED
        assert h.heddle_device_errors(ctx) == 0
    finally:
        h.heddle_destroy(ctx)


def test_tiling_full_size_sampled(h, W, oracle_mod):
    """moe48 at its full 1e6 candidates in one call: every OK candidate and
    a random sample of the rest against the oracle."""
    w = W.make_workload("moe48", seed=0)
    got = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, *_experts(w))
    assert got["errors"] == 0
    rng = np.random.default_rng(5)
    ok = np.nonzero(got["status"] == 0)[0]
    idx = np.unique(np.concatenate([ok, rng.choice(w.cands["S"].shape[0], 4000, replace=False)]))
    sub = G.take(w.cands, idx)
    ref = _oracle(oracle_mod, w).price(sub, threads=8, tiling=True)
    G.assert_same(got, ref, idx=idx, what="moe48 full tiled")
    okr = ref["status"] == 0
    assert (got["tiling"][:, idx][:, okr] == ref["tiling"][:, okr]).all()
