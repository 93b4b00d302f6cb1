"""Micro-batch-size fill (§5.3) on the GPU through the C ABI against the
oracle's fill: bit-exact T, bottleneck, n_dp, status, bounds and chosen
size on seeded workloads with per-size profiles, and with the synthetic
formula on scaled FLOPs and messages."""

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


def _same(gpu, orc, what):
    G.assert_same(gpu, orc, what=what)
    bad = np.nonzero(gpu["mbs"] != orc["mbs"])[0]
    assert bad.size == 0, "%s mbs differs at %d candidates, first %s: gpu %s oracle %s" % (
        what, bad.size, bad[:5], gpu["mbs"][bad[:5]], orc["mbs"][bad[:5]])


@pytest.mark.parametrize("name,n", [("tiny_ext", None), ("dense32", 5003), ("dense80", 1201),
                                    ("moe48", 4001), ("stress128", 611)])
@pytest.mark.parametrize("levels", [2, 4])
@pytest.mark.parametrize("search", [0, 1], ids=["auto", "general"])
def test_mbs_parity_profiles(h, W, oracle_mod, name, n, levels, search):
    w = W.make_workload(name, seed=1, n=n)
    prof = W.mbs_profiles(w, levels, seed=1)
    ref = oracle_mod.price_mbs(w.cluster, w.model, w.cands, levels, prof, threads=8)
    got = G.price_mbs_gpu(h, w.cluster, w.model, w.cands, levels, prof, search=search)
    assert got["errors"] == 0
    _same(got, ref, "%s levels %d" % (name, levels))


@pytest.mark.parametrize("name,n", [("dense32", 4003), ("moe48", 3001), ("stress128", 503)])
def test_mbs_parity_formula(h, W, oracle_mod, name, n):
    w = W.make_workload(name, seed=2, n=n)
    ref = oracle_mod.price_mbs(w.cluster, w.model, w.cands, 3, None, threads=8)
    got = G.price_mbs_gpu(h, w.cluster, w.model, w.cands, 3, None)
    assert got["errors"] == 0
    _same(got, ref, "%s formula" % name)


def test_mbs_one_level_is_plain_pricing(h, W, oracle_mod):
    w = W.make_workload("dense32", seed=3, n=3001)
    got = G.price_mbs_gpu(h, w.cluster, w.model, w.cands, 1, None)
    plain = G.price_gpu(h, w.cluster, w.model, w.cands, bounds=True)
    for key in ("T", "bottleneck", "n_dp", "status", "bounds"):
        assert (got[key] == plain[key]).all(), key
    assert (got["mbs"] == 0).all()


def test_mbs_more_than_one_chunk(h, W, oracle_mod):
    """A batch above the 2^20-candidate chunk: sampled candidates of both
    chunks against the oracle."""
    n = (1 << 20) + 70001
    w = W.make_workload("dense32", seed=4, n=n)
    prof = W.mbs_profiles(w, 3, seed=4)
    got = G.price_mbs_gpu(h, w.cluster, w.model, w.cands, 3, prof, bounds=False)
    rng = np.random.default_rng(4)
    idx = np.sort(np.concatenate([rng.choice(1 << 20, 1500, replace=False),
                                  (1 << 20) + rng.choice(70001, 1500, replace=False)]))
    ref = oracle_mod.price_mbs(w.cluster, w.model, G.take(w.cands, idx), 3, prof, threads=8, bounds=False)
    sub = {k: got[k][idx] for k in ("T", "bottleneck", "n_dp", "status", "mbs")}
    sub["bounds"] = None
    _same(sub, ref, "two chunks")
    assert (got["mbs"] > 0).any()


def test_mbs_call_errors(h, W):
    import torch
    w = W.make_workload("tiny", seed=0)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(int(w.cands["S"].shape[0]))
        with pytest.raises(h.HeddleError) as e:
            h.heddle_price_mbs(ctx, h.make_candidates(dc), h.make_results(res))
        assert e.value.status == 2  # E_STATE
        with pytest.raises(h.HeddleError) as e:
            h.heddle_load_mbs(ctx, h.MAX_MBS_LEVELS + 1)
        assert e.value.status == 3  # E_LIMIT
        bad = W.mbs_profiles(w, 2)
        bad[1][0, 0, 0] = float("nan")
        with pytest.raises(h.HeddleError) as e:
            h.heddle_load_mbs(ctx, 2, bad)
        assert e.value.status == 1  # E_ARG
        h.heddle_load_mbs(ctx, 2, W.mbs_profiles(w, 2))
        h.heddle_price_mbs(ctx, h.make_candidates(dc), h.make_results(res))
        torch.cuda.synchronize()
        h.heddle_load_mbs(ctx, 0)
        with pytest.raises(h.HeddleError):
            h.heddle_price_mbs(ctx, h.make_candidates(dc), h.make_results(res))
    finally:
        h.heddle_destroy(ctx)
