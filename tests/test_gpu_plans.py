"""Multi-template plans (Algorithm 1) on the GPU through the C ABI against
the oracle's plan pricing: bit-exact per-template T, bottleneck, n_dp and
status (the plan's degree on the GPUs earlier templates left, SKIPPED past
the end), templates placed and the summed throughput (IEEE double)."""

import json
import os

import numpy as np
import pytest

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


def price_plans_gpu(h, cluster, model, plans, search=None, bounds=False):
    import torch
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, cluster)
        h.heddle_load_model(ctx, model)
        if search is not None:
            h.heddle_set_search(ctx, search)
        dp = h.plans_to_device(plans)
        n = int(plans["n_tmpl"].shape[0])
        pr = h.alloc_plan_results(n, len(dp["slots"]), bounds=bounds)
        h.heddle_price_plans(ctx, dp, pr)
        torch.cuda.synchronize()
        out = {k: np.stack([h.results_to_numpy(r)[k] for r in pr["slots"]]) for k in ("T", "bottleneck", "n_dp", "status")}
        out["placed"] = pr["placed"].cpu().numpy()
        out["thr"] = pr["thr"].cpu().numpy()
        out["errors"] = h.heddle_device_errors(ctx)
        if bounds:
            out["bounds"] = [r["bounds"].cpu().numpy() for r in pr["slots"]]
        return out
    finally:
        h.heddle_destroy(ctx)


def _same(got, ref, what):
    for k in ("T", "bottleneck", "n_dp", "status"):
        bad = np.argwhere(got[k] != ref[k])
        assert bad.size == 0, "%s %s differs at %s: gpu %s oracle %s" % (
            what, k, bad[:5].tolist(), got[k][tuple(bad[0])], ref[k][tuple(bad[0])])
    assert (got["placed"] == ref["placed"]).all(), what
    bad = np.nonzero(got["thr"] != ref["thr"])[0]
    assert bad.size == 0, "%s thr differs at %s: %s vs %s" % (what, bad[:5], got["thr"][bad[:3]], ref["thr"][bad[:3]])


@pytest.mark.parametrize("name,n", [("tiny", 300), ("dense32", 4001), ("dense80", 1501), ("moe48", 4001),
                                    ("stress128", 701)])
@pytest.mark.parametrize("seed", [0, 1])
def test_plans_parity(h, W, oracle_mod, name, n, seed):
    w = W.make_workload(name, seed=seed, n=n)
    plans = W.make_plans(w, n, 4, seed=seed)
    ref = oracle_mod.Oracle(w.cluster, w.model).price_plans(plans)
    got = price_plans_gpu(h, w.cluster, w.model, plans)
    assert got["errors"] == 0
    _same(got, ref, "%s plans" % name)
    assert (ref["placed"] >= 1).any()
    if name in ("dense32", "dense80", "stress128"):  # later templates priced on what is left
        assert (ref["placed"] >= 2).any()


@pytest.mark.parametrize("search", [1, 3], ids=["general", "distribute"])
def test_plans_other_split_modes(h, W, oracle_mod, search):
    w = W.make_workload("dense32", seed=5, n=2001)
    plans = W.make_plans(w, 2001, 3, seed=5)
    orc = oracle_mod.Oracle(w.cluster, w.model)
    if search == 3:
        orc.set_split("distribute")
    ref = orc.price_plans(plans)
    got = price_plans_gpu(h, w.cluster, w.model, plans, search=search)
    _same(got, ref, "dense32 search %d" % search)


def test_plans_bounds(h, W, oracle_mod):
    """With bound planes requested: an OK template keeps the split of its
    standalone price (the oracle's, slot by slot), every other template's
    planes are zero (slots that no plan reaches included)."""
    w = W.make_workload("dense32", seed=3, n=3001)
    plans = W.make_plans(w, 3001, 3, seed=3)
    ref = oracle_mod.Oracle(w.cluster, w.model).price_plans(plans)
    got = price_plans_gpu(h, w.cluster, w.model, plans, bounds=True)
    _same(got, ref, "dense32 plans with bounds")
    orc = oracle_mod.Oracle(w.cluster, w.model)
    for t in range(3):
        alone = orc.price({"S": np.ascontiguousarray(plans["S"][t]), "M": np.ascontiguousarray(plans["M"][t]),
                           "code": np.ascontiguousarray(plans["code"][t])}, bounds=True)
        b = got["bounds"][t]
        ok = got["status"][t] == 0
        assert ok.any() and (~ok).any(), t
        assert (b[:, ok] == alone["bounds"][:, ok]).all(), t
        assert (b[:, ~ok] == 0).all(), t


def test_plans_hand_cases(h, W):
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "hand_plans.json")
    d = json.load(open(path))
    cl = d["cluster"]
    cluster = W.make_cluster(cl["tflops"], cl["mem_bytes"], cl["intra_bw"], [tuple(x) for x in cl["nodes"]])
    model = W.make_model(d["flops"], 0, 0, 0, 0, 0, 0)
    import pin_checks as PC
    for case in d["cases"]:
        got = price_plans_gpu(h, cluster, model, PC._plans_from(case["templates"], case["n_tmpl"], W))
        e = case["expect"]
        assert got["status"][:, 0].tolist() == e["status"], case["name"]
        assert got["n_dp"][:, 0].tolist() == e["n_dp"], case["name"]
        assert got["T"][:, 0].tolist() == e["T"], case["name"]
        assert int(got["placed"][0]) == e["placed"], case["name"]
        assert float(got["thr"][0]) == e["thr"], case["name"]


def test_plans_limits(h, W):
    import torch
    w = W.make_workload("tiny", seed=0)
    plans = W.make_plans(w, 10, 2, seed=0)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        dp = h.plans_to_device(plans)
        pr = h.alloc_plan_results(10, 2)
        h.heddle_price_plans(ctx, dp, pr)
        torch.cuda.synchronize()
        big = W.make_cluster([1000.0], [10**11], [10**11], [(0, 72, 10**10)])
        h.heddle_load_cluster(ctx, big)
        with pytest.raises(h.HeddleError) as e:
            h.heddle_price_plans(ctx, dp, pr)
        assert e.value.status == 3  # E_LIMIT: a node above the plan limit
    finally:
        h.heddle_destroy(ctx)
