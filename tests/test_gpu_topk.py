"""heddle_topk over seeded result planes built to stress its filters:
throughput rising along the batch (so an unsorted slice keeps producing new
bests), near-ties whose float keys n*M / T are equal while their exact order
is not, exact ties in throughput with other factors, and a second call into
the filled state; k on both sides of 32 (the first pass that sets a floor
runs for k <= 32 while the state is not full).  Compared with the oracle's
top-k of everything offered so far."""

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

KS = (1, 16, 32, 33, 64)


def _planes(n, seed, n_top):
    rng = np.random.default_rng(seed)
    # T falls along the batch: n*M / T rises with the index
    T = (np.int64(1) << 40) - np.arange(n, dtype=np.int64) * 4096 - rng.integers(0, 4096, n)
    ndp = np.full(n, 8, np.uint16)
    M = np.full(n, 64, np.uint16)
    status = np.where(rng.random(n) < 0.7, 0, rng.integers(1, 4, n)).astype(np.uint8)
    # the best n_top: T within 2 of 2^39 (equal float keys, distinct exact
    # keys), a third of them at twice T with twice n (exact ties)
    top = rng.choice(n, n_top, replace=False)
    T[top] = (np.int64(1) << 39) + rng.integers(0, 3, n_top)
    status[top] = 0
    twin = top[: n_top // 3]
    T[twin] *= 2
    ndp[twin] = 16
    return {"T": T, "n_dp": ndp, "M": M, "status": status}


def _run_topk(h, ctx, planes, base, state):
    import torch
    n = int(planes["T"].shape[0])
    dev = {key: torch.from_numpy(v.view(np.int16) if v.dtype == np.uint16 else v).cuda()
           for key, v in planes.items()}
    c = h.heddle_candidates(dev["M"].data_ptr(), dev["M"].data_ptr(), dev["M"].data_ptr(), n, n, 1, 0, base)
    r = h.heddle_results(dev["T"].data_ptr(), dev["T"].data_ptr(), dev["n_dp"].data_ptr(),
                         dev["status"].data_ptr(), None)
    h.heddle_topk(ctx, c, r, state)
    torch.cuda.synchronize()
    return h.read_topk_state(state)


def _same_state(got, exp, what):
    assert got["count"] == exp["count"], what
    n = exp["count"]
    for key in ("idx", "T", "nM"):
        assert np.array_equal(np.asarray(got[key])[:n], np.asarray(exp[key])[:n]), "%s: %s" % (what, key)


@pytest.mark.parametrize("k", KS)
@pytest.mark.parametrize("n_top", (10, 150))
def test_topk_rising_batch_and_near_ties(heddle_lib, oracle_mod, k, n_top):
    import torch
    h = heddle_lib
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    first = _planes(300_001, 3 + k, n_top)
    second = _planes(123_457, 7 + k, n_top)
    state = h.alloc_topk_state()
    ctx = h.heddle_create(0)
    try:
        h.heddle_topk_reset(ctx, state, k)
        got1 = _run_topk(h, ctx, first, 0, state)
        exp1 = oracle_mod.topk({key: first[key] for key in ("T", "n_dp", "status")}, first["M"], k)
        assert exp1["count"] == k
        _same_state(got1, exp1, "k=%d, %d best, first call" % (k, n_top))
        got2 = _run_topk(h, ctx, second, first["T"].shape[0], state)
        union = {key: np.concatenate([first[key], second[key]]) for key in ("T", "n_dp", "status", "M")}
        exp2 = oracle_mod.topk({key: union[key] for key in ("T", "n_dp", "status")}, union["M"], k)
        _same_state(got2, exp2, "k=%d, %d best, second call" % (k, n_top))
    finally:
        h.heddle_destroy(ctx)
