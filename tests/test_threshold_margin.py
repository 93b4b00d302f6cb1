"""The top-k threshold of a pricing call (a float word below the running
state's k-th key n*M / T) drops an entry only when its float key falls
below the threshold.  The threshold is fl(fl(fl(nM_k) / fl(T_k)) * (1 - 2^-16))
and an entry's key fl(fl(nM) / fl(T)), every operation IEEE single
precision with round-to-nearest as the kernels compute them.  Dropping
must be exact: an entry whose exact key is at least the k-th's is never
below the threshold.  Checked here on the host in float32 for random,
near-tied and extreme keys (numpy may convert a 64-bit integer through
float64, rounding twice, which stays within the same error bound)."""

import numpy as np

MARGIN = np.float32(1.0 - 1.0 / 65536.0)


def fkey(nM, T):
    return np.float32(nM).astype(np.float32) / np.float32(T).astype(np.float32)


def threshold(nM, T):
    return (fkey(nM, T) * MARGIN).astype(np.float32)


def exact_ge(nMa, Ta, nMb, Tb):
    """a's key >= b's key, exactly (Python integers)."""
    return [int(x) * int(tb) >= int(y) * int(ta) for x, ta, y, tb in zip(nMa, Ta, nMb, Tb)]


def check(nMa, Ta, nMb, Tb):
    ge = np.array(exact_ge(nMa, Ta, nMb, Tb))
    kept = fkey(nMa, Ta) >= threshold(nMb, Tb)
    # every entry at least as good as the k-th entry b is kept
    assert kept[ge].all()
    return int(ge.sum())


def test_random_keys():
    rng = np.random.default_rng(0)
    n = 200000
    nMa = rng.integers(1, 1 << 32, n, dtype=np.uint64)
    nMb = rng.integers(1, 1 << 32, n, dtype=np.uint64)
    Ta = rng.integers(1, 1 << 62, n, dtype=np.uint64)
    Tb = rng.integers(1, 1 << 62, n, dtype=np.uint64)
    assert check(nMa, Ta, nMb, Tb) > 0


def test_near_ties():
    rng = np.random.default_rng(1)
    n = 200000
    Tb = rng.integers(1 << 20, 1 << 62, n, dtype=np.uint64)
    nMb = rng.integers(1, 1 << 32, n, dtype=np.uint64)
    # a: the same key, one ns faster, one more micro-batch, or a scaled copy
    d = rng.integers(0, 3, n)
    Ta = np.where(d == 0, Tb - 1, np.where(d == 1, Tb, Tb * 2 // 2))
    nMa = np.where(d == 1, np.minimum(nMb + 1, (1 << 32) - 1), nMb).astype(np.uint64)
    assert check(nMa, Ta.astype(np.uint64), nMb, Tb) == n


def test_extremes():
    vals_T = np.array([1, 2, 3, (1 << 24) - 1, 1 << 24, (1 << 24) + 1, (1 << 53) + 1, (1 << 62) - 1,
                       (1 << 63) - 1], dtype=np.uint64)
    vals_nM = np.array([1, 2, 255, 65535, 65536, (1 << 24) + 1, (1 << 32) - 1], dtype=np.uint64)
    A = [(m, t) for m in vals_nM for t in vals_T]
    nMa = np.array([a[0] for a in A for _ in A], dtype=np.uint64)
    Ta = np.array([a[1] for a in A for _ in A], dtype=np.uint64)
    nMb = np.array([b[0] for _ in A for b in A], dtype=np.uint64)
    Tb = np.array([b[1] for _ in A for b in A], dtype=np.uint64)
    assert check(nMa, Ta, nMb, Tb) > 0


def test_margin_is_not_too_loose():
    """The margin keeps extra entries only within 2^-15 of the k-th key."""
    rng = np.random.default_rng(2)
    n = 100000
    nMb = rng.integers(1, 1 << 32, n, dtype=np.uint64)
    Tb = rng.integers(1, 1 << 62, n, dtype=np.uint64)
    thr = threshold(nMb, Tb).astype(np.float64)
    exact = nMb.astype(np.float64) / Tb.astype(np.float64)
    assert (thr <= exact).all()
    assert (thr >= exact * (1 - 2.0 ** -15)).all()
