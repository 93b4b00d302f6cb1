"""The paper's own layer split (search mode DISTRIBUTE, §5.3 "Layer split
and DP degree") on the GPU through the C ABI against the oracle's same
rule: bit-exact T, bottleneck, n_dp, status, bounds and top-k."""

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


@pytest.mark.parametrize("name,n", [("tiny", None), ("tiny_ext", None), ("dense32", 6007), ("dense80", 1531),
                                    ("moe48", 6011), ("stress128", 613)])
@pytest.mark.parametrize("seed", [0, 1])
def test_distribute_parity(h, W, oracle_mod, name, n, seed):
    w = W.make_workload(name, seed=seed, n=n)
    ref = oracle_mod.Oracle(w.cluster, w.model).set_split("distribute").price(w.cands, threads=8)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, search=h.SEARCH_DISTRIBUTE)
    assert got["errors"] == 0
    assert got["search"] == h.SEARCH_DISTRIBUTE
    G.assert_same(got, ref, what="%s distribute" % name)
    tk = oracle_mod.topk(ref, w.cands["M"], 16)
    assert got["topk"]["idx"].tolist() == tk["idx"].tolist()


def test_distribute_hand_cases(h, W, oracle_mod):
    """The hand-worked cases of the paper's rule, on the GPU."""
    import json
    import os
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_distribute.json")
    for case in json.load(open(path))["cases"]:
        nt = len(case["tflops"])
        cluster = W.make_cluster(case["tflops"], case["mem_bytes"], [300 * 10**9] * nt,
                                 [tuple(x) for x in case["nodes"]])
        model = W.make_model(case["flops"], 0, case["state_bytes"], case["act_bytes"], 0, 0, 0)
        cands = W.from_structures([[tuple(s) for s in case["stages"]]], [4])
        got = G.price_gpu(h, cluster, model, cands, search=h.SEARCH_DISTRIBUTE)
        e = case["expect"]
        assert int(got["status"][0]) == e["status"], case["name"]
        assert int(got["T"][0]) == e["T"], case["name"]
        assert int(got["bottleneck"][0]) == e["bottleneck"], case["name"]
        if e["bounds"] is not None:
            S = len(case["stages"])
            assert got["bounds"][: S + 1, 0].tolist() == e["bounds"], case["name"]


def test_distribute_never_beats_the_exact_bottleneck(h, W):
    w = W.make_workload("dense80", seed=3, n=20011)
    exact = G.price_gpu(h, w.cluster, w.model, w.cands, bounds=False)
    dist = G.price_gpu(h, w.cluster, w.model, w.cands, bounds=False, search=h.SEARCH_DISTRIBUTE)
    ok = dist["status"] == 0
    assert ok.sum() > 100
    assert (exact["status"][ok] == 0).all()
    assert (dist["bottleneck"][ok] >= exact["bottleneck"][ok]).all()
