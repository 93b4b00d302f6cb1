"""heddle_topk_noalloc: the top-k merge for callers that cannot allocate
device memory (no context, scratch in a fixed device array).  It must leave
the same state as heddle_topk, on two calls in a row that merge two batches
into one state.  Kept in its own file, collected last."""

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def test_noalloc_topk_matches_topk_on_two_calls(heddle_lib):
    import torch
    from paper_2609_34244_gb300 import workloads as W
    h = heddle_lib
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    w = W.make_workload("moe48", seed=0, n=300_000)
    n = w.n
    ctx = h.heddle_create(0)
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(n)
        ref_state, na_state = h.alloc_topk_state(), h.alloc_topk_state()
        h.heddle_topk_reset(ctx, ref_state, 64)
        h.heddle_topk_reset(ctx, na_state, 64)
        half = n // 2
        for lo, hi in ((0, half), (half, n)):  # two calls in a row into one state
            c = h.make_candidates(dc, lo, hi)
            r = h.make_results(res, lo, hi)
            h.heddle_price_candidates(ctx, c, r)
            h.heddle_topk(ctx, c, r, ref_state)
            h.heddle_topk_noalloc(c, r, na_state)
            torch.cuda.synchronize()
            ref = h.read_topk_state(ref_state)
            got = h.read_topk_state(na_state)
            assert ref["count"] > 0
            for key in ("count", "k"):
                assert got[key] == ref[key]
            for key in ("idx", "T", "nM"):
                assert np.array_equal(got[key], ref[key]), key
        assert h.heddle_device_errors(ctx) == 0
    finally:
        h.heddle_destroy(ctx)
    # a batch above the fixed scratch is rejected with E_LIMIT, not run
    big = h.heddle_candidates(dc["S"].data_ptr(), dc["M"].data_ptr(), dc["code"].data_ptr(),
                              h.TOPK_NOALLOC_MAX_N + 1, h.TOPK_NOALLOC_MAX_N + 1, 12, 0, 0)
    with pytest.raises(h.HeddleError) as e:
        h.heddle_topk_noalloc(big, h.make_results(res), na_state)
    assert e.value.status == 3
