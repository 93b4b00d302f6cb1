"""heddle_topk_noalloc: the top-k merge for callers that cannot allocate
device memory (no context, scratch in a fixed device array).

Checked against the oracle's top-k and against heddle_topk, on two calls in a
row that merge two batches into one state, for k = 1, 16 and 64; on priced
candidates and on seeded synthetic result planes: a batch of exactly the
maximum size, a ragged batch over more than 16 slices, slices without any
OK candidate, and ties in throughput.  Kept in its own file, collected
last."""

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

KS = (1, 16, 64)


def _same_state(got, exp, what):
    assert got["count"] == exp["count"], what
    n = exp["count"]
    for key in ("idx", "T", "nM"):
        assert np.array_equal(np.asarray(got[key])[:n], np.asarray(exp[key])[:n]), "%s: %s" % (what, key)


@pytest.mark.parametrize("k", KS)
def test_noalloc_topk_matches_oracle_and_topk_on_two_calls(heddle_lib, oracle_mod, k):
    import torch
    from paper_2609_34244_gb300 import workloads as W
    h = heddle_lib
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    w = W.make_workload("moe48", seed=0, n=300_000)
    n = w.n
    ref_all = oracle_mod.Oracle(w.cluster, w.model).price(w.cands, threads=8, bounds=False)
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(n)
        ref_state, na_state = h.alloc_topk_state(), h.alloc_topk_state()
        h.heddle_topk_reset(ctx, ref_state, k)
        h.heddle_topk_reset(ctx, na_state, k)
        half = n // 2
        for lo, hi in ((0, half), (half, n)):  # two calls in a row into one state
            c = h.make_candidates(dc, lo, hi)  # global indices: base lo
            r = h.make_results(res, lo, hi)
            h.heddle_price_candidates(ctx, c, r)
            h.heddle_topk(ctx, c, r, ref_state)
            h.heddle_topk_noalloc(c, r, na_state)
            torch.cuda.synchronize()
            got = h.read_topk_state(na_state)
            _same_state(got, h.read_topk_state(ref_state), "k=%d vs heddle_topk" % k)
            seen = {key: ref_all[key][:hi] for key in ("T", "n_dp", "status")}
            exp = oracle_mod.topk(seen, w.cands["M"][:hi], k)
            assert exp["count"] > 0
            _same_state(got, exp, "k=%d vs oracle after [0, %d)" % (k, hi))
        assert h.heddle_device_errors(ctx) == 0
    finally:
        h.heddle_destroy(ctx)
    # a batch above the fixed scratch is rejected with E_LIMIT, not run
    big = h.heddle_candidates(dc["S"].data_ptr(), dc["M"].data_ptr(), dc["code"].data_ptr(),
                              h.TOPK_NOALLOC_MAX_N + 1, h.TOPK_NOALLOC_MAX_N + 1, 12, 0, 0)
    with pytest.raises(h.HeddleError) as e:
        h.heddle_topk_noalloc(big, h.make_results(res), na_state)
    assert e.value.status == 3


def _synthetic(n, seed, empty_slices):
    """Seeded result planes: about 30% OK, no OK candidate in the listed
    slices of 65,536, and a run of exact throughput ties near the top."""
    rng = np.random.default_rng(seed)
    T = rng.integers(10**6, 10**12, n, dtype=np.int64)
    ndp = rng.integers(1, 65, n).astype(np.uint16)
    M = rng.integers(1, 513, n).astype(np.uint16)
    status = np.where(rng.random(n) < 0.3, 0, rng.integers(1, 4, n)).astype(np.uint8)
    # ties: candidates with equal n*M / T, the best throughput of the batch
    tie = rng.choice(n, 40, replace=False)
    status[tie] = 0
    T[tie] = 1000
    ndp[tie] = 8
    M[tie] = 500
    T[tie[:10]] = 2000   # the same ratio with other factors
    ndp[tie[:10]] = 16
    for s in empty_slices:
        status[s * 65536:(s + 1) * 65536] = 1
    return {"T": T, "n_dp": ndp, "M": M, "status": status}


def _run_noalloc(h, planes, base, state):
    import torch
    n = int(planes["T"].shape[0])
    dev = {key: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).cuda()
           for key, v in planes.items()}
    c = h.heddle_candidates(dev["M"].data_ptr(), dev["M"].data_ptr(), dev["M"].data_ptr(), n, n, 1, 0, base)
    r = h.heddle_results(dev["T"].data_ptr(), dev["T"].data_ptr(), dev["n_dp"].data_ptr(),
                         dev["status"].data_ptr(), None)
    h.heddle_topk_noalloc(c, r, state)
    torch.cuda.synchronize()
    return h.read_topk_state(state)


@pytest.mark.parametrize("k", KS)
def test_noalloc_topk_synthetic_maximum_and_ragged(heddle_lib, oracle_mod, k):
    import torch
    h = heddle_lib
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    # exactly the maximum (64 slices) with empty slices, then a ragged batch
    # of 17 slices (the last partly filled, slice 16 with no OK candidate)
    first = _synthetic(h.TOPK_NOALLOC_MAX_N, 11 + k, empty_slices=(0, 3, 17, 40, 41, 42, 63))
    second = _synthetic(16 * 65536 + 12345, 29 + k, empty_slices=(5, 16))
    state = h.alloc_topk_state()
    ctx = h.heddle_create(0)
    try:
        h.heddle_topk_reset(ctx, state, k)
        torch.cuda.synchronize()
    finally:
        h.heddle_destroy(ctx)
    got1 = _run_noalloc(h, first, 0, state)
    exp1 = oracle_mod.topk({"T": first["T"], "n_dp": first["n_dp"], "status": first["status"]}, first["M"], k)
    _same_state(got1, exp1, "k=%d maximum batch" % k)
    got2 = _run_noalloc(h, second, h.TOPK_NOALLOC_MAX_N, state)
    union = {key: np.concatenate([first[key], second[key]]) for key in ("T", "n_dp", "status", "M")}
    exp2 = oracle_mod.topk({"T": union["T"], "n_dp": union["n_dp"], "status": union["status"]}, union["M"], k)
    _same_state(got2, exp2, "k=%d after the ragged batch" % k)
    # a batch whose every slice is empty leaves the state as it was
    none_ok = _synthetic(3 * 65536 + 7, 5, empty_slices=(0, 1, 2, 3))
    got3 = _run_noalloc(h, none_ok, 2 * h.TOPK_NOALLOC_MAX_N, state)
    _same_state(got3, exp2, "k=%d after a batch with no OK candidate" % k)
