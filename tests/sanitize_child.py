"""Child process of ``test_sanitizers.py``: runs under LD_PRELOAD of the
AddressSanitizer runtime, with the instrumented oracle (HEDDLE_ORACLE_LIB)
or the instrumented CUDA library (HEDDLE_LIB) loaded instead of the plain
builds.

  python sanitize_child.py oracle OUT.npz   -- every oracle entry point on small
                                               seeded workloads; results saved
  python sanitize_child.py capi             -- the C ABI's host-side checks that
                                               run without a device
"""

import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def oracle_run(out_path):
    from oracle import oracle as O
    from paper_2609_34244_gb300 import workloads as W
    res = {}
    for name, n in (("tiny", None), ("tiny_ext", None), ("dense32", 600), ("dense80", 400), ("moe48", 600),
                    ("stress128", 300)):
        w = W.make_workload(name, seed=1, n=n)
        orc = O.Oracle(w.cluster, w.model)
        r = orc.price(w.cands, threads=2, bounds=True)
        for k in ("T", "bottleneck", "n_dp", "status", "bounds"):
            res["%s_%s" % (name, k)] = r[k]
        t = O.topk(r, w.cands["M"], 16)
        res[name + "_topk"] = t["idx"]
        orc.set_split("distribute")
        d = orc.price(w.cands, threads=2, bounds=True)
        res[name + "_dist_T"] = d["T"]
        res[name + "_dist_bounds"] = d["bounds"]
        q = orc.tables()
        res[name + "_q"] = q["q"]
        res[name + "_p2p"] = q["p2p"]
    w = W.make_workload("moe16", seed=2, n=300)
    orc = O.Oracle(w.cluster, w.model).set_experts(w.model["expert_state_bytes"], w.model["expert_param_bytes"])
    r = orc.price(w.cands, threads=2, bounds=True, tiling=True)
    res["moe16_tiled_T"] = r["T"]
    res["moe16_tiling"] = r["tiling"]
    w = W.make_workload("stress128", seed=3, n=2000)
    plans = W.make_plans(w, 200, 4, seed=3)
    p = O.Oracle(w.cluster, w.model).price_plans(plans)
    res["plans_T"] = p["T"]
    res["plans_thr"] = p["thr"]
    w = W.make_workload("dense32", seed=4, n=300)
    m = O.price_mbs(w.cluster, w.model, w.cands, 3, W.mbs_profiles(w, 3, seed=4), threads=2)
    res["mbs_T"] = m["T"]
    res["mbs"] = m["mbs"]
    rng = np.random.default_rng(5)
    raw = []
    for _ in range(50):
        S, L = int(rng.integers(1, 6)), int(rng.integers(1, 13))
        P = np.concatenate([np.zeros((S, 1), np.int64), np.cumsum(rng.integers(0, 9, (S, L)), axis=1)], axis=1)
        c = rng.integers(0, 5, S)
        Wm = np.concatenate([np.zeros((S, 1), np.int64), np.cumsum(rng.integers(0, 5, (S, L)), axis=1)], axis=1)
        cap = rng.integers(3, 30, S)
        r = O.partition_raw(P, c, Wm, cap)
        raw.append(-1 if r is None else r[0])
    res["raw_B"] = np.asarray(raw, np.int64)
    res["replicas"] = np.asarray([O.replicas([8, 4, 2, 2], [2, 4]), O.replicas([8, 8], [8, 1, 1])], np.int64)
    np.savez(out_path, **res)


def capi_run():
    from paper_2609_34244_gb300 import heddle as h
    L = h.load_library()
    import ctypes as C
    # no context: every call that needs one refuses it
    assert L.heddle_load_cluster(None, None, 0, None, 0) == h.E_ARG
    assert L.heddle_load_model(None, None, 0, 0, 0, None) == h.E_ARG
    assert L.heddle_price_candidates(None, None, None, None) == h.E_ARG
    assert L.heddle_topk(None, None, None, None, None) == h.E_ARG
    assert L.heddle_set_chunk(None, 1) == h.E_ARG
    assert L.heddle_set_search(None, 0) == h.E_ARG
    h.heddle_destroy(None)
    assert isinstance(L.heddle_last_error(None), bytes)
    # the allocation-free top-k checks its arguments before any device call
    c = h.heddle_candidates(None, None, None, -1, 0, 1, 0, 0)
    r = h.heddle_results(None, None, None, None, None)
    assert L.heddle_topk_noalloc(C.byref(c), C.byref(r), None, None) == h.E_ARG
    assert L.heddle_topk_noalloc(None, C.byref(r), None, None) == h.E_ARG
    c = h.heddle_candidates(1, 1, 1, h.TOPK_NOALLOC_MAX_N + 1, h.TOPK_NOALLOC_MAX_N + 1, 1, 0, 0)
    assert L.heddle_topk_noalloc(C.byref(c), C.byref(r), C.c_void_p(16), None) == h.E_LIMIT
    c = h.heddle_candidates(1, 0, 1, 5, 5, 1, 0, 0)
    assert L.heddle_topk_noalloc(C.byref(c), C.byref(r), C.c_void_p(16), None) == h.E_ARG
    # without a device, creating a context fails cleanly with *out NULL
    out = C.c_void_p(1234)
    st = L.heddle_create(C.byref(out), 0)
    assert st == h.E_CUDA and not out.value, (st, out.value)
    print("capi ok")


if __name__ == "__main__":
    if sys.argv[1] == "oracle":
        oracle_run(sys.argv[2])
    else:
        capi_run()
