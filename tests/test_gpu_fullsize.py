"""Full-size workloads in the benchmark's launch configuration, compared with
the oracle on every candidate.

The oracle prices every candidate of each full-size workload here (all host
threads; the 1e7-candidate stress workload takes a minute or two on 16
cores), once per session.  Its results must also reproduce the digests in
``golden/fullsize_oracle.json`` (written by the oracle alone), which pins the
seeded inputs and the oracle's own output on this host to the ones stored.
The GPU path -- one pricing call over all candidates in chunks of 1e6, as
the benchmark times it, and separately one price + top-k call per 1e6 batch
-- must then match the oracle on every field of every candidate and its
top-16 must equal the oracle's top-16 over the whole set, for the
equal-layer search (auto) and the general search."""

import json
import os

import numpy as np
import pytest

import fullsize_common as F
import gpu_helpers as G

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "fullsize_oracle.json")
_ORACLE = {}


def _golden():
    with open(GOLDEN) as f:
        return json.load(f)


def _oracle_full(oracle_mod, name, n):
    """The workload and the oracle's results over all of it (cached)."""
    if name not in _ORACLE:
        from paper_2609_34244_gb300 import workloads as W
        w = W.make_workload(name, seed=F.SEED, n=n)
        ref = oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=os.cpu_count() or 1, bounds=False)
        top = oracle_mod.topk(ref, w.cands["M"], F.TOPK)
        _ORACLE.clear()  # one full-size workload held at a time
        _ORACLE[name] = (w, ref, top)
    return _ORACLE[name]


@pytest.mark.parametrize("path", ["bench", "batched"])
@pytest.mark.parametrize("search", [0, 1], ids=["auto", "general"])
@pytest.mark.parametrize("name,n", F.FULL_SIZES)
def test_full_size(heddle_lib, oracle_mod, name, n, search, path):
    import torch
    assert torch.cuda.is_available()
    h = heddle_lib
    w, ref, top = _oracle_full(oracle_mod, name, n)
    gold = _golden()[F.key(name, n)]
    assert F.input_digest(w.cands) == gold["inputs_sha256"], "seeded inputs differ from the stored ones"
    assert F.field_digests(ref) == gold["fields_sha256"], "the oracle on this host differs from the stored run"
    assert [int(x) for x in top["idx"]] == gold["topk"]["idx"]
    if path == "bench":
        # one call over every candidate, priced in 1e6 chunks pipelined over
        # the work streams and merged in order (the benchmark's step)
        got = G.price_gpu(h, w.cluster, w.model, w.cands, k=F.TOPK, bounds=False, search=search, fused=True,
                          chunk=1_000_000)
    else:
        got = G.price_gpu(h, w.cluster, w.model, w.cands, k=F.TOPK, bounds=False, batch=1_000_000,
                          search=search)
    assert got["errors"] == 0
    if search == 1:
        assert got["search"] == h.SEARCH_GENERAL
    G.assert_same(got, ref, what="%s %s" % (name, path))
    assert F.field_digests(got) == gold["fields_sha256"]
    tk = got["topk"]
    assert tk["count"] == top["count"]
    assert tk["idx"].tolist() == top["idx"].tolist()
    assert tk["T"].tolist() == top["T"].tolist()
    assert tk["nM"].tolist() == top["nM"].tolist()


@pytest.mark.parametrize("thread_min", [0, 2**31 - 1], ids=["thread", "warp"])
def test_full_size_general_routes(heddle_lib, oracle_mod, thread_min):
    """moe48 at full size with the general search's routing forced each way
    (by default its few single-fit entries go to the warp kernel)."""
    h = heddle_lib
    name, n = "moe48", 1_000_000
    w, ref, top = _oracle_full(oracle_mod, name, n)
    got = G.price_gpu(h, w.cluster, w.model, w.cands, k=F.TOPK, bounds=False, search=h.SEARCH_GENERAL,
                      fused=True, chunk=1_000_000, thread_min=thread_min)
    assert got["errors"] == 0
    G.assert_same(got, ref, what="moe48 thread_min %d" % thread_min)
    assert got["topk"]["idx"].tolist() == top["idx"].tolist()


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
