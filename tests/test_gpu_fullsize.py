"""Full-size workloads in the benchmark's launch configuration (device-resident
batches of at most 1e6 candidates priced and merged into one top-k state):
every sampled candidate bit-exact against the oracle, the top-k equal to an
exact host top-k of the GPU's own per-candidate outputs, and every top-k
entry re-priced by the oracle."""

import numpy as np
import pytest

import gpu_helpers as G

pytestmark = pytest.mark.gpu

FULL = [("dense32", 100_000, None), ("dense80", 1_000_000, 4000), ("moe48", 1_000_000, 4000),
        ("stress128", 10_000_000, 300)]


@pytest.mark.parametrize("search", [0, 1], ids=["auto", "general"])
@pytest.mark.parametrize("name,n,per_batch_sample", FULL)
def test_full_size(heddle_lib, oracle_mod, name, n, per_batch_sample, search):
    import torch
    from paper_2609_34244_gb300 import workloads as W
    assert torch.cuda.is_available()
    h = heddle_lib
    w = W.make_workload(name, seed=0, n=n)
    batch = 1_000_000
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, bounds=False, batch=batch, search=search)
    assert got["errors"] == 0
    orc = oracle_mod.Oracle(w.cluster, w.model)
    rng = np.random.default_rng(123)
    if per_batch_sample is None:
        idx = np.arange(n)
    else:
        idx = np.concatenate([lo + rng.choice(min(batch, n - lo), per_batch_sample, replace=False)
                              for lo in range(0, n, batch)])
    sub = W.make_cands(w.cands["S"][idx], w.cands["M"][idx], np.ascontiguousarray(w.cands["code"][:, idx]))
    ref = orc.price(sub, threads=16, bounds=False)
    G.assert_same(got, ref, idx=idx, what=name)
    # top-k of the GPU outputs, computed exactly on the host
    ok = np.nonzero(got["status"] == 0)[0]
    nM = got["n_dp"][ok].astype(np.int64) * w.cands["M"][ok].astype(np.int64)
    exp = G.exact_topk(ok, got["T"][ok], nM, 16)
    assert got["topk"]["idx"].tolist() == [e[0] for e in exp]
    # and every top-k entry priced again by the oracle
    ti = got["topk"]["idx"]
    tsub = W.make_cands(w.cands["S"][ti], w.cands["M"][ti], np.ascontiguousarray(w.cands["code"][:, ti]))
    tref = orc.price(tsub, bounds=False)
    assert (tref["T"] == got["topk"]["T"]).all()
    assert (tref["n_dp"].astype(np.uint32) * w.cands["M"][ti].astype(np.uint32) == got["topk"]["nM"]).all()


def test_one_call_larger_than_the_worklist(heddle_lib, oracle_mod):
    """A single pricing call of 1.2e6 candidates (more than one 2^20-candidate
    worklist chunk) with bounds, checked on a sample."""
    import torch
    from paper_2609_34244_gb300 import workloads as W
    h = heddle_lib
    n = 1_200_000
    w = W.make_workload("dense32", seed=7, n=n)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, bounds=True)
    assert got["errors"] == 0
    rng = np.random.default_rng(9)
    idx = np.sort(np.concatenate([rng.choice(n, 3000, replace=False), np.arange((1 << 20) - 50, (1 << 20) + 50)]))
    sub = W.make_cands(w.cands["S"][idx], w.cands["M"][idx], np.ascontiguousarray(w.cands["code"][:, idx]))
    ref = oracle_mod.Oracle(w.cluster, w.model).price(sub, threads=16)
    G.assert_same(got, ref, idx=idx, what="dense32 1.2e6")


def _sample(n, batch, per_batch, seed):
    rng = np.random.default_rng(seed)
    return np.concatenate([lo + rng.choice(min(batch, n - lo), min(per_batch, n - lo), replace=False)
                           for lo in range(0, n, batch)])


@pytest.mark.parametrize("name,n,per_batch_sample", [("dense80", 1_000_000, 3000), ("moe48", 1_000_000, 3000),
                                                     ("stress128", 10_000_000, 200)])
def test_full_size_distribute(heddle_lib, oracle_mod, name, n, per_batch_sample):
    """The paper's split mode at full size in 1e6 batches, sampled."""
    from paper_2609_34244_gb300 import workloads as W
    h = heddle_lib
    w = W.make_workload(name, seed=0, n=n)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, bounds=False, batch=1_000_000,
                      search=h.SEARCH_DISTRIBUTE)
    assert got["errors"] == 0
    idx = _sample(n, 1_000_000, per_batch_sample, 321)
    ref = oracle_mod.Oracle(w.cluster, w.model).set_split("distribute").price(G.take(w.cands, idx), threads=16,
                                                                            bounds=False)
    G.assert_same(got, ref, idx=idx, what=name + " distribute")
    ok = np.nonzero(got["status"] == 0)[0]
    nM = got["n_dp"][ok].astype(np.int64) * w.cands["M"][ok].astype(np.int64)
    exp = G.exact_topk(ok, got["T"][ok], nM, 16)
    assert got["topk"]["idx"].tolist() == [e[0] for e in exp]


@pytest.mark.parametrize("name,n,per_batch_sample", [("dense80", 1_000_000, 2000), ("stress128", 10_000_000, 150)])
def test_full_size_mbs(heddle_lib, oracle_mod, name, n, per_batch_sample):
    """The micro-batch-size fill (four sizes, per-size profiles) at full size
    in 1e6 batches, sampled."""
    from paper_2609_34244_gb300 import workloads as W
    h = heddle_lib
    w = W.make_workload(name, seed=0, n=n)
    prof = W.mbs_profiles(w, 4, seed=0)
    got = G.price_mbs_gpu(h, w.cluster, w.model, w.cands, 4, prof, bounds=False, batch=1_000_000)
    assert got["errors"] == 0
    idx = _sample(n, 1_000_000, per_batch_sample, 654)
    ref = oracle_mod.price_mbs(w.cluster, w.model, G.take(w.cands, idx), 4, prof, threads=16, bounds=False)
    sub = {k: got[k][idx] for k in ("T", "bottleneck", "n_dp", "status", "mbs")}
    sub["bounds"] = None
    G.assert_same(sub, ref, what=name + " fill")
    assert (sub["mbs"] == ref["mbs"]).all()
