"""Child process of ``test_gpu_checked.py``: prices seeded workloads with the
bounds-checked build of the library (HEDDLE_LIB) in every search mode and
compares every result with the oracle; any raised device flag fails."""

import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(HERE))
sys.path.insert(0, HERE)


def main():
    import gpu_helpers as G
    from oracle import oracle as O
    from paper_2609_34244_gb300 import heddle as h, workloads as W
    assert os.environ.get("HEDDLE_LIB", "").endswith("libheddle_checked.so")
    cases = (("tiny_ext", None), ("dense32", 30011), ("dense80", 20011), ("moe48", 30011), ("stress128", 150001))
    for name, n in cases:
        w = W.make_workload(name, seed=3, n=n)
        for mode, split, tmin in ((h.SEARCH_AUTO, "minmax", None), (h.SEARCH_GENERAL, "minmax", None),
                                  (h.SEARCH_GENERAL, "minmax", 0), (h.SEARCH_DISTRIBUTE, "distribute", None)):
            ref = O.Oracle(w.cluster, w.model).set_split(split).price(w.cands, threads=8)
            for fused in (False, True):
                got = G.price_gpu(h, w.cluster, w.model, w.cands, k=16, search=mode, fused=fused, chunk=65536,
                                  thread_min=tmin)
                assert got["errors"] == 0, "%s mode %d: device flags %#x" % (name, mode, got["errors"])
                G.assert_same(got, ref, what="%s mode %d fused %s" % (name, mode, fused))
                exp = O.topk(ref, w.cands["M"], 16)
                assert got["topk"]["idx"].tolist() == exp["idx"].tolist(), (name, mode)
    # plans: the per-slot SKIPPED mask and the walk
    import test_gpu_plans as TP
    for name in ("dense32", "stress128"):
        w = W.make_workload(name, seed=4, n=3001)
        plans = W.make_plans(w, 3001, 4, seed=4)
        ref = O.Oracle(w.cluster, w.model).price_plans(plans)
        got = TP.price_plans_gpu(h, w.cluster, w.model, plans, bounds=True)
        assert got["errors"] == 0, "%s plans: device flags %#x" % (name, got["errors"])
        TP._same(got, ref, "%s plans" % name)
    w = W.make_workload("moe16", seed=2, n=20011)
    ref = O.Oracle(w.cluster, w.model).set_experts(w.model["expert_state_bytes"], w.model["expert_param_bytes"]) \
        .price(w.cands, threads=8)
    got = G.price_tiled_gpu(h, w.cluster, w.model, w.cands, w.model["expert_state_bytes"],
                            w.model["expert_param_bytes"])
    assert got["errors"] == 0
    G.assert_same(got, ref, what="moe16 tiled")
    print("checked ok")


if __name__ == "__main__":
    main()
