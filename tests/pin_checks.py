"""Pins for the CPU oracle: each check compares the oracle against something
other than itself -- hand-worked values (``tests/golden``), brute-force
enumeration, closed forms and invariants.  Every check raises
AssertionError on a mismatch.  ``test_oracle_pins.py`` runs them; the
mutation test runs them against deliberately broken copies of the oracle and
requires each copy to fail at least one.
"""

from __future__ import annotations

import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
UNIT = 10**6  # hand examples count costs in units scaled to nanoseconds


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _workloads():
    from paper_2609_34244_gb300 import workloads as W
    return W


# ---------------------------------------------------------------- helpers

def tables_from_scales(layers, scales, c, mem_layers=None, mem_cap=None):
    """Raw stage tables: stage s costs scale_s * sum(layers) + c_s; memory
    prefix of ``mem_layers`` (same for every stage) against ``mem_cap``."""
    base = np.concatenate([[0], np.cumsum(np.asarray(layers, dtype=np.int64))])
    P = np.stack([base * int(k) for k in scales])
    if mem_layers is None:
        W = np.zeros_like(P)
        cap = np.zeros(len(scales), np.int64)
    else:
        m = np.concatenate([[0], np.cumsum(np.asarray(mem_layers, dtype=np.int64))])
        W = np.stack([m for _ in scales])
        cap = np.asarray(mem_cap, dtype=np.int64)
    return P, np.asarray(c, dtype=np.int64), W, cap


def brute_partition(P, c, W, cap):
    """Every contiguous split into S non-empty stages, in lexicographic order
    of the boundary vector; returns (B*, first optimal boundaries) or None."""
    S, L1 = P.shape
    L = L1 - 1
    best = None
    for cut in itertools.combinations(range(1, L), S - 1):
        a = (0,) + cut + (L,)
        ok = True
        worst = 0
        for s in range(S):
            i, j = a[s], a[s + 1]
            if W[s][j] - W[s][i] > cap[s]:
                ok = False
                break
            worst = max(worst, int(P[s][j] - P[s][i] + c[s]))
        if ok and (best is None or worst < best[0]):
            best = (worst, list(a))
    return best


def brute_replicas(node_gpus, groups, limit=64):
    """Largest n such that n copies of ``groups`` can be assigned to nodes
    (exhaustive backtracking over assignments)."""
    def fits(items, caps):
        items = sorted(items, reverse=True)
        caps = list(caps)

        def rec(t):
            if t == len(items):
                return True
            seen = set()
            for b in range(len(caps)):
                if caps[b] >= items[t] and caps[b] not in seen:
                    seen.add(caps[b])
                    caps[b] -= items[t]
                    if rec(t + 1):
                        return True
                    caps[b] += items[t]
            return False
        return rec(0)

    n = 0
    while n < limit and fits(list(groups) * (n + 1), node_gpus):
        n += 1
    return n


def oracle_for(O, case):
    W = _workloads()
    cl = case["cluster"]
    cluster = W.make_cluster(cl["tflops"], cl["mem_bytes"], cl["intra_bw"],
                             [tuple(x) for x in cl["nodes"]])
    m = case["model"]
    L = len(m["flops"])
    model = W.make_model(m["flops"], m["param_bytes"], m["state_bytes"], m["act_bytes"],
                         m["ar_bytes"], m["a2a_bytes"], m["boundary_bytes"], moe=m["moe"])
    cands = W.from_structures([[tuple(s) for s in cd["stages"]] for cd in case["cands"]],
                              [cd["M"] for cd in case["cands"]])
    return O.Oracle(cluster, model), cands, L


# ------------------------------------------------------------------- pins

def check_hand_partitions(O):
    """Hand-worked PartitionLayers examples (golden/hand_partition.json)."""
    for case in _load("hand_partition.json")["cases"]:
        P, c, W, cap = tables_from_scales(case["layers"], case["scales"], case["c"],
                                          case.get("mem_layers"), case.get("mem_cap"))
        got = O.partition_raw(P * UNIT, c * UNIT, W, cap)
        if case["Bstar"] is None:
            assert got is None, case["name"]
            continue
        assert got is not None, case["name"]
        assert got[0] == case["Bstar"] * UNIT, (case["name"], got)
        assert got[1] == case["bounds"], (case["name"], got)


def check_hand_pricing(O):
    """Hand-worked end-to-end prices (golden/hand_pricing.json)."""
    for case in _load("hand_pricing.json")["cases"]:
        orc, cands, L = oracle_for(O, case)
        r = orc.price(cands)
        for c, exp in enumerate(case["expect"]):
            name = "%s cand %d" % (case["name"], c)
            assert int(r["status"][c]) == exp["status"], (name, r["status"][c])
            assert int(r["n_dp"][c]) == exp["n_dp"], (name, r["n_dp"][c])
            assert int(r["T"][c]) == exp["T"], (name, r["T"][c])
            assert int(r["bottleneck"][c]) == exp["bottleneck"], (name, r["bottleneck"][c])
            S = int(cands["S"][c])
            if exp["bounds"] is not None:
                assert r["bounds"][: S + 1, c].tolist() == exp["bounds"], (name, r["bounds"][:, c])
        if "topk_order" in case:
            tk = O.topk(r, cands["M"], len(case["expect"]))
            assert tk["idx"].tolist() == case["topk_order"], (case["name"], tk)


def check_brute_force_partition(O, trials=400, seed=1234):
    """Oracle DP == exhaustive enumeration of every contiguous split on small
    random heterogeneous instances (memory caps that sometimes bind)."""
    rng = np.random.default_rng(seed)
    for t in range(trials):
        S = int(rng.integers(1, 6))
        L = int(rng.integers(S, 13))
        layers = rng.integers(0, 50, L)
        scales = rng.integers(1, 6, S)
        c = rng.integers(0, 30, S) if rng.random() < 0.7 else np.zeros(S, np.int64)
        c[-1] = 0
        P = np.stack([np.concatenate([[0], np.cumsum(layers * k)]) for k in scales]).astype(np.int64)
        # per-stage memory tables (different weights per stage, as in-flight counts differ)
        mw = rng.integers(0, 10, L)
        W = np.stack([np.concatenate([[0], np.cumsum(mw * (1 + (S - s) % 3))]) for s in range(S)])
        tot = W[:, -1]
        cap = (tot * rng.uniform(0.2, 1.2, S)).astype(np.int64) if rng.random() < 0.6 else tot
        exp = brute_partition(P, c, W, cap)
        got = O.partition_raw(P, c, W, cap)
        if exp is None:
            assert got is None, (t, got)
        else:
            assert got is not None, (t, exp)
            assert got[0] == exp[0] and got[1] == exp[1], (t, S, L, got, exp)


def check_closed_forms(O, seed=7):
    """S = 1 is the serial sum; uniform unit costs give B* = ceil(L/S) with the
    leftmost optimal split; identical stages with no P2P and no memory limit
    are the textbook linear-partition problem: B* >= ceil(P[L]/S) and B* does
    not increase when a stage is added."""
    rng = np.random.default_rng(seed)
    for L in range(1, 20):
        layers = rng.integers(1, 100, L)
        P, c, W, cap = tables_from_scales(layers, [1], [0])
        assert O.partition_raw(P, c, W, cap) == (int(layers.sum()), [0, L])
        for S in range(1, L + 1):
            P, c, W, cap = tables_from_scales(np.ones(L, np.int64), [1] * S, [0] * S)
            B, a = O.partition_raw(P, c, W, cap)
            assert B == math.ceil(L / S), (L, S, B)
            # leftmost: every boundary as small as the remainder allows
            for s in range(1, S):
                assert a[s] == max(s, L - (S - s) * B), (L, S, a)
    for trial in range(60):
        L = int(rng.integers(2, 30))
        layers = rng.integers(0, 1000, L)
        prev = None
        for S in range(1, min(L, 8) + 1):
            P, c, W, cap = tables_from_scales(layers, [1] * S, [0] * S)
            B, a = O.partition_raw(P, c, W, cap)
            assert B >= math.ceil(layers.sum() / S)
            assert B >= layers.max()
            if prev is not None:
                assert B <= prev, (layers, S, B, prev)
            prev = B


def check_replicas(O, trials=150, seed=99):
    """First-fit-decreasing replication count == exhaustive placement search
    on small clusters; plus hand cases."""
    assert O.replicas([8, 4], [4, 2, 2]) == 1
    assert O.replicas([3, 3], [2, 1]) == 2
    assert O.replicas([3, 3], [2, 2]) == 1
    assert O.replicas([3, 3], [2, 2, 2]) == 0
    assert O.replicas([8], [1]) == 8
    assert O.replicas([4, 4, 4, 4], [4, 4]) == 2
    assert O.replicas([2, 2], [4]) == 0
    rng = np.random.default_rng(seed)
    for t in range(trials):
        nodes = [int(x) for x in rng.integers(1, 6, int(rng.integers(1, 4)))]
        mx = max(nodes)
        opts = [g for g in (1, 2, 4) if g <= mx]
        groups = [int(rng.choice(opts)) for _ in range(int(rng.integers(1, 4)))]
        exp = brute_replicas(nodes, groups, limit=sum(nodes))
        assert O.replicas(nodes, groups) == exp, (nodes, groups, exp)


def check_quantiser(O):
    """Nearest-nanosecond rounding with halves away from zero, via an explicit
    profile (the per-(type, degree, layer) cost entry of the paper's cost
    model, §5.2)."""
    W = _workloads()
    vals = [(2.0e-3, 2_000_000), (0.0, 0), (2.0**-12, 244_141), (2.0**-11, 488_281)]
    # j * 2^-10 s is exactly j * 976562.5 ns: for odd j an exact tie, rounded
    # away from zero; one ulp below the tie rounds down
    for j in (1, 3, 5, 1001):
        x = j * 2.0**-10
        assert x * 1e9 == j * 976562.5
        vals.append((x, j * 976562 + (j + 1) // 2))
        vals.append((math.nextafter(x, 0.0), j * 976562 + (j - 1) // 2))
    L = len(vals)
    prof = np.zeros((1, 4, L))
    prof[0, :, :] = [v for v, _ in vals]
    cluster = W.make_cluster([1000.0], [10**12], [10**11], [(0, 8, 10**10)])
    model = W.make_model(np.ones(L), 1, 1, 1, 0, 0, 0, profile_s=prof)
    q = O.Oracle(cluster, model).tables()["q"]
    for l, (v, exp) in enumerate(vals):
        assert (q[0, :, l] == exp).all(), (l, v, q[0, :, l], exp)


def check_layer_cost_formula(O):
    """Per-layer cost entries of the synthetic profile: compute, TP all-reduce
    and EP all-to-all terms on round numbers worked out by hand."""
    W = _workloads()
    # type 0: 1000 TFLOPS, intra 300 GB/s, two 4-GPU nodes with 12.5 GB/s NICs
    cluster = W.make_cluster([1000.0], [10**12], [300 * 10**9],
                             [(0, 4, 12_500_000_000), (0, 4, 12_500_000_000)])
    # layer 0: 1e12 FLOPs, 75 MB all-reduce; layer 1: 2e12 FLOPs, 100 MB all-to-all
    model = W.make_model([1e12, 2e12], 1, 1, 1, [75_000_000, 0], [0, 100_000_000], 0, moe=True)
    q = O.Oracle(cluster, model).tables()["q"][0]
    # k=1: 1 ms, 2 ms
    assert q[0].tolist() == [1_000_000, 2_000_000]
    # k=2: 0.5 ms + 4*(2*1/2)*75e6/3e11 s = 0.5 + 1 = 1.5 ms; 1 ms + 4*(1/2)*1e8/3e11 s = 1 + 0.6667 ms
    assert q[1].tolist() == [1_500_000, 1_666_667]
    # k=4: 0.25 + 4*(2*3/4)*75e6/3e11 = 0.25 + 1.5 = 1.75 ms; 0.5 + 4*(3/4)*1e8/3e11 = 0.5 + 1 = 1.5 ms
    assert q[2].tolist() == [1_750_000, 1_500_000]
    # k=8 exceeds the 4-GPU node: NIC 12.5 GB/s.  0.125 + 4*(2*7/8)*75e6/1.25e10 = 0.125 + 42 ms;
    # 0.25 + 4*(7/8)*1e8/1.25e10 = 0.25 + 28 ms
    assert q[3].tolist() == [42_125_000, 28_250_000]


def check_invariants(O, seed=3):
    """On random workloads: T >= M * B*; T = M*P[L] + g for S = 1; bounds
    strictly increasing from 0 to L; outputs follow a permutation of the
    candidates; the top-k of shards merged equals the top-k of the whole."""
    W = _workloads()
    for name, n in (("dense32", 600), ("moe48", 600), ("dense80", 150)):
        w = W.make_workload(name, seed=seed, n=n)
        orc = O.Oracle(w.cluster, w.model)
        r = orc.price(w.cands)
        tab = orc.tables()
        ok = r["status"] == 0
        M = w.cands["M"].astype(np.int64)
        assert (r["T"][ok] >= M[ok] * r["bottleneck"][ok]).all()
        assert (r["T"][~ok] == -1).all() and (r["bottleneck"][~ok] == -1).all()
        L = w.meta["L"]
        for c in np.nonzero(ok)[0]:
            S = int(w.cands["S"][c])
            a = r["bounds"][: S + 1, c].astype(int)
            assert a[0] == 0 and a[-1] == L and (np.diff(a) > 0).all()
            if S == 1:
                code = int(w.cands["code"][0, c])
                PL = int(tab["P"][code & 7, (code >> 3) & 3, L])
                assert r["bottleneck"][c] == PL
                if r["n_dp"][c] == 1:
                    assert r["T"][c] == int(M[c]) * PL
        assert (np.diff(tab["P"], axis=2) >= 0).all()
        perm = np.random.default_rng(seed).permutation(w.n)
        pc = {"S": w.cands["S"][perm], "M": w.cands["M"][perm],
              "code": np.ascontiguousarray(w.cands["code"][:, perm])}
        rp = orc.price(pc)
        for key in ("T", "bottleneck", "n_dp", "status"):
            assert (rp[key] == r[key][perm]).all(), key
        full = O.topk(r, w.cands["M"], 16)
        pool = []
        for lo in range(0, w.n, 97):
            hi = min(w.n, lo + 97)
            sub = {k: r[k][lo:hi] for k in ("T", "n_dp", "status")}
            part = O.topk(sub, w.cands["M"][lo:hi], 16, base_index=lo)
            pool += zip(part["idx"].tolist(), part["T"].tolist(), part["nM"].tolist())
        # merge the shard lists by exact throughput n*M/T, then smaller index
        pool.sort(key=lambda e: (-Fraction(e[2], e[1]), e[0]))
        assert [e[0] for e in pool[:16]] == full["idx"].tolist()
        pk = O.topk(rp, pc["M"], 16)
        assert [int(perm[i]) for i in pk["idx"]] == full["idx"].tolist()


def check_status_rules(O):
    """Masked structures are INVALID (§5.1 masks): reserved bits, unknown type,
    S > L, S = 0, M = 0, TP degree above the largest node of a dense type."""
    W = _workloads()
    cluster = W.make_cluster([1000.0, 500.0], [10**12, 10**12], [10**11, 10**11],
                             [(0, 4, 10**10), (1, 2, 10**10)])
    model = W.make_model([1e12] * 3, 1, 1, 1, 0, 0, 0)
    orc = O.Oracle(cluster, model)
    S = np.array([1, 1, 1, 4, 0, 1, 1, 1, 2], np.uint8)
    M = np.array([1, 1, 1, 1, 1, 0, 1, 1, 1], np.uint16)
    code = np.zeros((4, 9), np.uint8)
    code[0] = [0x20, 2, 0, 0, 0, 0, int(W.encode(1, 2)), int(W.encode(0, 2)), 0]
    code[1, 8] = int(W.encode(1, 1))
    code[:, 3] = 0
    r = orc.price({"S": S, "M": M, "code": code})
    assert r["status"].tolist() == [3, 3, 0, 3, 3, 3, 3, 0, 0], r["status"]


def check_mbs_hand(O):
    """Hand-worked micro-batch-size fill (golden/hand_mbs.json, §5.3)."""
    W = _workloads()
    d = _load("hand_mbs.json")
    cl, m = d["cluster"], d["model"]
    L = m["L"]
    for case in d["cases"]:
        cluster = W.make_cluster(cl["tflops"], [case["mem_bytes"]], cl["intra_bw"],
                                 [tuple(x) for x in cl["nodes"]])
        model = W.make_model([m["flops"]] * L, m["param_bytes"], m["state_bytes"], m["act_bytes"],
                             m["ar_bytes"], m["a2a_bytes"], case.get("boundary_bytes", m["boundary_bytes"]))
        if case["level_ms"] is None:
            levels, profiles = case["levels"], None
        else:
            levels = len(case["level_ms"])
            profiles = [np.full((1, 4, L), ms / 1000.0) for ms in case["level_ms"]]
        cands = W.from_structures([[(0, 0), (0, 0)]], [case["M"]])
        r = O.price_mbs(cluster, model, cands, levels, profiles)
        e = case["expect"]
        name = case["name"]
        assert int(r["status"][0]) == e["status"], (name, r["status"][0])
        assert int(r["mbs"][0]) == e["mbs"], (name, r["mbs"][0])
        assert int(r["T"][0]) == e["T"], (name, r["T"][0])
        assert int(r["bottleneck"][0]) == e["bottleneck"], (name, r["bottleneck"][0])
        if e["bounds"] is not None:
            assert r["bounds"][:3, 0].tolist() == e["bounds"], (name, r["bounds"][:3, 0])


def check_mbs_properties(O, seed=11):
    """Properties of the fill on seeded workloads with per-size profiles:
    stored activations grow with the size at fixed micro-batches per
    iteration, so a candidate that does not fit at the base size fits at no
    size; a one-size fill is the plain price; the chosen size divides M."""
    W = _workloads()
    for name, n in (("dense32", 3000), ("moe48", 3000)):
        w = W.make_workload(name, seed=seed, n=n)
        prof = W.mbs_profiles(w, 3, seed=seed)
        plain = O.Oracle(w.cluster, O.level_model(w.model, 0, prof[0])).price(w.cands)
        one = O.price_mbs(w.cluster, w.model, w.cands, 1, prof[:1])
        for k in ("T", "bottleneck", "n_dp", "status"):
            assert (one[k] == plain[k]).all(), (name, k)
        r = O.price_mbs(w.cluster, w.model, w.cands, 3, prof)
        assert not ((plain["status"] == O.OOM) & (r["status"] == O.OK)).any(), name
        # each larger size on its own: a candidate that is not OK at the
        # base size is OK at none (the library prices only the base size's
        # OK candidates at the larger sizes)
        M0 = np.asarray(w.cands["M"], np.int64)
        for i in (1, 2):
            ci = dict(w.cands)
            ci["M"] = np.where(M0 % (1 << i) == 0, M0 >> i, 0).astype(np.uint16)
            li = O.Oracle(w.cluster, O.level_model(w.model, i, prof[i])).price(ci)
            assert not ((plain["status"] != O.OK) & (li["status"] == O.OK)).any(), (name, i)
            assert (li["status"][plain["status"] == O.OOM] != O.OK).all(), (name, i)
        assert ((r["status"] == O.OK) | (r["status"] == plain["status"])).all(), name
        M = np.asarray(w.cands["M"], np.int64)
        assert ((M % (1 << r["mbs"].astype(np.int64))) == 0).all(), name
        ok = r["status"] == O.OK
        assert (r["T"][ok & (plain["status"] == O.OK)] <= plain["T"][ok & (plain["status"] == O.OK)]).all(), name
        if name == "dense32":  # 11% OK: some candidate gains from a larger size
            assert (r["mbs"] > 0).any(), (name, "a larger size wins somewhere")


def check_distribute_hand(O):
    """Hand-worked prices under the paper's own split rule
    (golden/hand_distribute.json, §5.3)."""
    W = _workloads()
    for case in _load("hand_distribute.json")["cases"]:
        nt = len(case["tflops"])
        cluster = W.make_cluster(case["tflops"], case["mem_bytes"], [300 * 10**9] * nt,
                                 [tuple(x) for x in case["nodes"]])
        L = len(case["flops"])
        model = W.make_model(case["flops"], 0, case["state_bytes"], case["act_bytes"], 0, 0, 0)
        cands = W.from_structures([[tuple(s) for s in case["stages"]]], [4])
        S = len(case["stages"])
        for mode, e in (("distribute", case["expect"]), ("minmax", case.get("minmax"))):
            if e is None:
                continue
            r = O.Oracle(cluster, model).set_split(mode).price(cands)
            name = "%s (%s)" % (case["name"], mode)
            assert int(r["status"][0]) == e["status"], (name, r["status"][0])
            assert int(r["T"][0]) == e["T"], (name, r["T"][0])
            assert int(r["bottleneck"][0]) == e["bottleneck"], (name, r["bottleneck"][0])
            if e["bounds"] is not None and mode == "distribute":
                assert r["bounds"][: S + 1, 0].tolist() == e["bounds"], (name, r["bounds"][:, 0])


def check_distribute_properties(O, seed=5):
    """The paper's rule against the exact split on seeded workloads: it
    fits only where some split fits, and its bottleneck is never below the
    min-max bottleneck B*; with equal layers, equal speeds and ample memory
    it is the equal-count split."""
    W = _workloads()
    for name, n in (("dense32", 2000), ("moe48", 2000), ("stress128", 400)):
        w = W.make_workload(name, seed=seed, n=n)
        exact = O.Oracle(w.cluster, w.model).price(w.cands)
        dist = O.Oracle(w.cluster, w.model).set_split("distribute").price(w.cands)
        okd = dist["status"] == O.OK
        assert (exact["status"][okd] == O.OK).all(), name
        assert (dist["bottleneck"][okd] >= exact["bottleneck"][okd]).all(), name
        same = dist["status"] != O.OK
        assert (dist["status"][same & (exact["status"] != O.OK)] == exact["status"][same & (exact["status"] != O.OK)]).all()
        if name != "moe48":  # moe48 is 1% OK even under the exact split
            assert okd.sum() > 0, name
        # the split precedes the DP degree (Algorithm 1): gradient bytes,
        # which only the gradient term sees, cannot change it
        m0 = dict(w.model)
        m0["param_bytes"] = np.zeros_like(np.asarray(w.model["param_bytes"]))
        d0 = O.Oracle(w.cluster, m0).set_split("distribute").price(w.cands)
        assert (d0["status"] == dist["status"]).all(), name
        assert (d0["bottleneck"] == dist["bottleneck"]).all(), name
        assert (d0["bounds"] == dist["bounds"]).all(), name
    cluster = W.make_cluster([1000.0], [10**13], [10**11], [(0, 8, 10**10)])
    model = W.make_model([1e12] * 10, 0, 0, 0, 0, 0, 0)
    cands = W.from_structures([[(0, 0)] * 3, [(0, 0)] * 4], [8, 8])
    r = O.Oracle(cluster, model).set_split("distribute").price(cands)
    assert r["bounds"][:4, 0].tolist() == [0, 4, 7, 10], r["bounds"][:, 0]
    assert r["bounds"][:5, 1].tolist() == [0, 3, 6, 8, 10], r["bounds"][:, 1]


def _plans_from(case_templates, n_tmpl, W):
    """Plan arrays for one plan from per-template stage lists."""
    tmax = len(case_templates)
    S = np.zeros((tmax, 1), np.uint8)
    M = np.full((tmax, 1), 4, np.uint16)
    code = np.zeros((tmax, 32, 1), np.uint8)
    for t, stages in enumerate(case_templates):
        S[t, 0] = len(stages)
        for s, (g, j) in enumerate(stages):
            code[t, s, 0] = int(W.encode(g, j))
    return {"n_tmpl": np.array([n_tmpl], np.uint8), "S": S, "M": M, "code": code}


def check_plans_hand(O):
    """Hand-worked multi-template plans (golden/hand_plans.json, Algorithm 1)."""
    W = _workloads()
    d = _load("hand_plans.json")
    cl = d["cluster"]
    cluster = W.make_cluster(cl["tflops"], cl["mem_bytes"], cl["intra_bw"], [tuple(x) for x in cl["nodes"]])
    model = W.make_model(d["flops"], 0, 0, 0, 0, 0, 0)
    orc = O.Oracle(cluster, model)
    for case in d["cases"]:
        r = orc.price_plans(_plans_from(case["templates"], case["n_tmpl"], W))
        e = case["expect"]
        name = case["name"]
        assert r["status"][:, 0].tolist() == e["status"], (name, r["status"][:, 0])
        assert r["n_dp"][:, 0].tolist() == e["n_dp"], (name, r["n_dp"][:, 0])
        assert r["T"][:, 0].tolist() == e["T"], (name, r["T"][:, 0])
        assert int(r["placed"][0]) == e["placed"], (name, r["placed"][0])
        assert float(r["thr"][0]) == e["thr"], (name, r["thr"][0])


def check_plans_properties(O, seed=2):
    """Plans on seeded workloads: a template priced first equals the plain
    price; ``placed`` counts the leading OK templates and later ones are
    skipped; the throughput adds up the placed templates' terms; a later
    template never has more replicas than it would on the whole cluster;
    the GPUs of the placed templates fit the cluster."""
    W = _workloads()
    for name, n in (("dense32", 300), ("moe48", 300), ("tiny", 200)):
        w = W.make_workload(name, seed=seed, n=n)
        plans = W.make_plans(w, n, 4, seed=seed)
        orc = O.Oracle(w.cluster, w.model)
        r = orc.price_plans(plans)
        first = orc.price({"S": plans["S"][0], "M": plans["M"][0], "code": plans["code"][0]})
        for k in ("T", "bottleneck", "n_dp", "status"):
            assert (r[k][0] == first[k]).all(), (name, k)
        tmax = plans["S"].shape[0]
        for c in range(n):
            p = int(r["placed"][c])
            st = r["status"][:, c]
            assert (st[:p] == O.OK).all(), (name, c)
            assert p == tmax or p == plans["n_tmpl"][c] or st[p] != O.OK, (name, c)
            assert (st[p + 1:] == O.SKIPPED).all() or (p < plans["n_tmpl"][c] and (st[p + 1:] == O.SKIPPED).all())
            acc = 0.0
            used = np.zeros(8, np.int64)
            for t in range(p):
                acc = acc + (float(int(r["n_dp"][t, c]) * int(plans["M"][t, c])) * 1e9) / float(r["T"][t, c])
                alone = orc.price({"S": plans["S"][t, c:c + 1], "M": plans["M"][t, c:c + 1],
                                   "code": plans["code"][t, :, c:c + 1]})
                assert int(r["n_dp"][t, c]) <= int(alone["n_dp"][0]), (name, c, t)
                for s in range(int(plans["S"][t, c])):
                    b = int(plans["code"][t, s, c])
                    used[b & 7] += int(r["n_dp"][t, c]) << ((b >> 3) & 3)
            assert acc == float(r["thr"][c]), (name, c)
            for g in range(len(w.cluster["tflops"])):
                assert used[g] <= int(w.cluster["node_gpus"][w.cluster["node_type"] == g].sum()), (name, c, g)


# ------------------------------------------------------------ expert tiling

def _tiled_oracle(O, W, case):
    cl = W.make_cluster(case["tflops"], case["mem_bytes"], case["intra_bw"], [tuple(x) for x in case["nodes"]])
    md = W.make_model(case["flops"], case["param_bytes"], case["state_bytes"], case["act_bytes"], case["ar_bytes"],
                      case["a2a_bytes"], case["boundary_bytes"], moe=True)
    return O.Oracle(cl, md).set_experts(case["expert_state"], case["expert_param"])


def check_tiling_hand(O):
    """Hand-worked prices with expert tiling (golden/hand_tiling.json, §5.3
    "Expert tiling"): ETP node bound, an EP group leaving a node, EDP
    memory replication, dense and expert gradient sync, re-selection
    against the whole iteration time."""
    W = _workloads()
    for case in _load("hand_tiling.json")["cases"]:
        o = _tiled_oracle(O, W, case)
        r = o.price(W.from_structures([[tuple(s) for s in case["stages"]]], [case["M"]]), tiling=True)
        S = len(case["stages"])
        e = case["expect"]
        got = {"status": int(r["status"][0]), "T": int(r["T"][0]), "bottleneck": int(r["bottleneck"][0]),
               "bounds": r["bounds"][: S + 1, 0].tolist(), "tiling": r["tiling"][:S, 0].tolist()}
        assert got == e, (case["name"], got)


def _tilings(j):
    """(le, lt, ld) of 2^j devices in slot order: EDP exponent ascending,
    then ETP exponent ascending."""
    return [(j - d - t, t, d) for d in range(j + 1) for t in range(j + 1 - d)]


def _tiled_instance(rng, W):
    nt = int(rng.integers(1, 3))
    nodes = [(g, int(rng.choice([2, 4])), int(rng.choice([1, 4, 10])) * 10**9)
             for g in range(nt) for _ in range(int(rng.integers(2, 7)))]
    cl = W.make_cluster(rng.uniform(0.5, 2.0, nt), rng.integers(20, 120, nt) * 10**9,
                        rng.choice([50, 100, 300], nt) * 10**9, nodes)
    L = int(rng.integers(3, 7))
    expert = rng.random(L) < 0.5
    es = np.where(expert, rng.integers(10, 80, L) * 10**9, 0)
    ep = np.where(expert, rng.integers(1, 50, L) * 10**8, 0)
    md = W.make_model(rng.uniform(1e9, 2e10, L), ep + rng.integers(1, 20, L) * 10**8,
                      es + rng.integers(1, 20, L) * 10**9, rng.integers(0, 5, L) * 10**9,
                      rng.integers(0, 5, L) * 10**7, np.where(expert, rng.integers(1, 20, L) * 10**7, 0),
                      int(rng.integers(0, 3)) * 10**7, moe=True)
    return cl, md, es, ep


def check_tiling_brute_force(O, trials=200, seed=77):
    """Tiled PartitionLayers and the re-selection against brute force on
    tiny random MoE instances: the split is the lexicographically smallest
    of those minimising the largest stage time when every stage takes its
    fastest fitting tiling (every split enumerated); T is the minimum over
    every combination of fitting tilings on that split; the reported
    tilings attain it, fit memory and keep ETP within a node; OOM exactly
    when no split fits under any tiling.  Stage costs come from the
    oracle's tiled tables (their values are pinned by the hand cases and by
    the untiled slot); gradient terms follow the stated formula."""
    W = _workloads()
    rng = np.random.default_rng(seed)
    seen_nontrivial = 0
    for _ in range(trials):
        cl, md, es, ep = _tiled_instance(rng, W)
        L = int(md["flops"].shape[0])
        nt = int(cl["tflops"].shape[0])
        structs = []
        for _c in range(10):
            S = int(rng.integers(1, min(3, L) + 1))
            structs.append([(int(rng.integers(0, nt)), int(rng.integers(0, 4))) for _s in range(S)])
        Ms = rng.choice([1, 2, 4, 8], len(structs))
        cands = W.from_structures(structs, Ms)
        o = O.Oracle(cl, md).set_experts(es, ep)
        r = o.price(cands, tiling=True)
        Pt = o.tiled_tables()["Pt"]
        tb = o.tables()
        maxn, inter, p2p = tb["maxnode"], tb["inter_bw"], tb["p2p"]
        st = np.concatenate([[0], np.cumsum(md["state_bytes"])])
        ex = np.concatenate([[0], np.cumsum(es)])
        ac = np.concatenate([[0], np.cumsum(md["act_bytes"])])
        pb = np.concatenate([[0], np.cumsum(md["param_bytes"])])
        eb = np.concatenate([[0], np.cumsum(ep)])
        for c, stages in enumerate(structs):
            S, M = len(stages), int(Ms[c])
            if int(r["status"][c]) not in (O.OK, O.OOM):
                continue
            n = int(r["n_dp"][c])
            opts, cs, caps = [], [], []
            for s, (g, j) in enumerate(stages):
                base = (0, 1, 4, 10)[j]
                opts.append([(base + i, le, lt, ld) for i, (le, lt, ld) in enumerate(_tilings(j))
                             if (1 << lt) <= maxn[g]])
                if s + 1 < S:
                    h, jn = stages[s + 1]
                    same = int(g == h and (1 << j) + (1 << jn) <= maxn[g])
                    cs.append(int(p2p[g, h, same]))
                else:
                    cs.append(0)
                caps.append(int(cl["mem_bytes"][g]) << j)

            def fits(s, i, e, o_):
                f = min(S - s, M)
                mem = (st[e] - st[i]) + ((1 << o_[3]) - 1) * (ex[e] - ex[i]) + f * (ac[e] - ac[i])
                return mem <= caps[s]

            def tcost(s, i, e, o_):
                return int(Pt[stages[s][0], o_[0], e] - Pt[stages[s][0], o_[0], i]) + cs[s]

            def gsync(s, i, e, o_):
                g, j = stages[s]
                Ge = int(eb[e] - eb[i])
                Gd = int(pb[e] - pb[i]) - Ge
                vol = (n - 1) * Gd + (n * (1 << o_[3]) - 1) * Ge
                if vol == 0:
                    return 0
                bw = int(cl["intra_bw"][g]) if (n == 1 and (1 << j) <= maxn[g]) else int(inter[g])
                return -((-2 * vol * 10**9) // (n * (1 << j) * bw))

            best, split = None, None
            for cut in itertools.combinations(range(1, L), S - 1):
                a = (0,) + cut + (L,)
                worst = 0
                for s in range(S):
                    ts = [tcost(s, a[s], a[s + 1], o_) for o_ in opts[s] if fits(s, a[s], a[s + 1], o_)]
                    if not ts:
                        worst = None
                        break
                    worst = max(worst, min(ts))
                if worst is not None and (best is None or worst < best):
                    best, split = worst, a
            if best is None:
                assert int(r["status"][c]) == O.OOM, (c, structs[c])
                continue
            assert int(r["status"][c]) == O.OK, (c, structs[c])
            assert tuple(r["bounds"][: S + 1, c].tolist()) == split, (c, split, r["bounds"][: S + 1, c])
            a = split
            choices = [[o_ for o_ in opts[s] if fits(s, a[s], a[s + 1], o_)] for s in range(S)]
            Tmin = None
            for combo in itertools.product(*choices):
                ts = [tcost(s, a[s], a[s + 1], combo[s]) for s in range(S)]
                gs = [gsync(s, a[s], a[s + 1], combo[s]) for s in range(S)]
                T = (M - 1) * max(ts) + sum(ts) + max(gs)
                Tmin = T if Tmin is None else min(Tmin, T)
            assert int(r["T"][c]) == Tmin, (c, int(r["T"][c]), Tmin)
            # the reported tilings: valid, fitting, and attaining T
            got = []
            for s in range(S):
                code = int(r["tiling"][s, c])
                le, lt = code & 3, code >> 2
                match = [o_ for o_ in choices[s] if o_[1] == le and o_[2] == lt]
                assert len(match) == 1, (c, s, code)
                got.append(match[0])
                seen_nontrivial += int(le != stages[s][1])
            ts = [tcost(s, a[s], a[s + 1], got[s]) for s in range(S)]
            gs = [gsync(s, a[s], a[s + 1], got[s]) for s in range(S)]
            assert (M - 1) * max(ts) + sum(ts) + max(gs) == Tmin, c
            assert max(ts) == int(r["bottleneck"][c]), c
    assert seen_nontrivial > 0


def check_tiling_reductions(O):
    """The untiled slot of every degree reproduces the untiled cost table
    bit for bit; a dense model with no expert bytes prices identically with
    tiling on and keeps the untiled tiling (EP over all devices) on every
    stage."""
    W = _workloads()
    for name in ("moe16", "moe48", "dense32"):
        w = W.make_workload(name, seed=3, n=600)
        es = w.model.get("expert_state_bytes")
        ep = w.model.get("expert_param_bytes")
        if es is None:
            es = ep = np.zeros(w.model["flops"].shape[0], np.int64)
        o = O.Oracle(w.cluster, w.model).set_experts(es, ep)
        P = o.tables()["P"]
        Pt = o.tiled_tables()["Pt"]
        for j in range(4):
            assert (Pt[:, (0, 1, 4, 10)[j], :] == P[:, j, :]).all(), (name, j)
        if name == "dense32":
            plain = O.Oracle(w.cluster, w.model).price(w.cands)
            tiled = o.price(w.cands, tiling=True)
            for k in ("T", "bottleneck", "n_dp", "status", "bounds"):
                assert (plain[k] == tiled[k]).all(), (name, k)
            ok = tiled["status"] == O.OK
            S = w.cands["S"][ok]
            live = np.arange(32)[:, None] < S[None, :]
            j = (w.cands["code"][:, ok] >> 3) & 3
            assert (tiled["tiling"][: j.shape[0], ok][live[: j.shape[0]]] == j[live[: j.shape[0]]]).all()


ALL_CHECKS = [
    check_hand_partitions,
    check_hand_pricing,
    check_brute_force_partition,
    check_closed_forms,
    check_replicas,
    check_quantiser,
    check_layer_cost_formula,
    check_invariants,
    check_status_rules,
    check_mbs_hand,
    check_mbs_properties,
    check_distribute_hand,
    check_distribute_properties,
    check_plans_hand,
    check_plans_properties,
    check_tiling_hand,
    check_tiling_brute_force,
    check_tiling_reductions,
]
