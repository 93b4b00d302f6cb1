"""ctypes wrapper around the CPU oracle (``heddle_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference arm are the only callers.  The product
path never imports this module.

The oracle takes the same seeded input dictionaries as the CUDA library (see
``paper_2609_34244_gb300.workloads``) and returns numpy arrays.
"""

from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "heddle_oracle.c")
HDR = os.path.join(HERE, "heddle_oracle.h")
# HEDDLE_ORACLE_LIB names a prebuilt library to load instead (the sanitizer
# test's instrumented build); it is then not rebuilt here
LIB = os.environ.get("HEDDLE_ORACLE_LIB") or os.path.join(HERE, "liboracle.so")

OK, OOM, NO_FIT, INVALID, SKIPPED = 0, 1, 2, 3, 4

_lib = None


def build(force: bool = False) -> str:
    """Compile ``liboracle.so`` with gcc (no fused multiply-add)."""
    if os.environ.get("HEDDLE_ORACLE_LIB"):
        return LIB
    newest = max(os.path.getmtime(SRC), os.path.getmtime(HDR))
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < newest:
        tmp = LIB + ".tmp%d" % os.getpid()
        subprocess.check_call(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
                               "-o", tmp, SRC, "-lpthread", "-lm"])
        os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(LIB)
        p = C.c_void_p
        L.orc_create.restype = p
        L.orc_create.argtypes = [C.c_int, p, p, p, C.c_int, p, p, p, C.c_int, p, p, p, p, p, p,
                                 C.c_int64, C.c_int, p, C.c_char_p]
        L.orc_destroy.argtypes = [p]
        L.orc_tables.argtypes = [p, p, p, p, p]
        L.orc_price.restype = C.c_int
        L.orc_price.argtypes = [p, C.c_int64, p, p, p, C.c_int64, C.c_int, p, p, p, p, p, C.c_int]
        L.orc_topk.restype = C.c_int
        L.orc_topk.argtypes = [C.c_int64, C.c_int64, p, p, p, p, C.c_int, p, p, p]
        L.orc_partition_raw.restype = C.c_int
        L.orc_partition_raw.argtypes = [C.c_int, C.c_int, p, p, p, p, p, p]
        L.orc_replicas.restype = C.c_int
        L.orc_replicas.argtypes = [C.c_int, p, C.c_int, p]
        L.orc_set_split.argtypes = [p, C.c_int]
        L.orc_set_experts.restype = C.c_int
        L.orc_set_experts.argtypes = [p, p, p, C.c_char_p]
        L.orc_tiled_tables.argtypes = [p, p, p]
        L.orc_price_tiled.restype = C.c_int
        L.orc_price_tiled.argtypes = [p, C.c_int64, p, p, p, C.c_int64, C.c_int, p, p, p, p, p, p, C.c_int]
        L.orc_price_plans.restype = C.c_int
        L.orc_price_plans.argtypes = [p, C.c_int64, C.c_int, p, p, p, p, C.c_int, p, p, p, p, p, p]
        _lib = L
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


class Oracle:
    """The oracle's cost model for one cluster and one model."""

    def __init__(self, cluster: dict, model: dict):
        L = lib()
        self._keep = []

        def arr(v, dt):
            a = np.ascontiguousarray(v, dtype=dt)
            self._keep.append(a)
            return a

        cl = {k: arr(cluster[k], dt) for k, dt in
              (("tflops", np.float64), ("mem_bytes", np.int64), ("intra_bw", np.int64),
               ("node_type", np.int32), ("node_gpus", np.int32), ("node_nic", np.int64))}
        md = {k: arr(model[k], dt) for k, dt in
              (("flops", np.float64), ("param_bytes", np.int64), ("state_bytes", np.int64),
               ("act_bytes", np.int64), ("ar_bytes", np.int64), ("a2a_bytes", np.int64))}
        prof = None if model.get("profile_s") is None else arr(model["profile_s"], np.float64)
        err = C.create_string_buffer(256)
        self.n_types = int(cl["tflops"].shape[0])
        self.L = int(md["flops"].shape[0])
        self._h = L.orc_create(self.n_types, _ptr(cl["tflops"]), _ptr(cl["mem_bytes"]),
                               _ptr(cl["intra_bw"]), int(cl["node_type"].shape[0]),
                               _ptr(cl["node_type"]), _ptr(cl["node_gpus"]), _ptr(cl["node_nic"]),
                               self.L, _ptr(md["flops"]), _ptr(md["param_bytes"]),
                               _ptr(md["state_bytes"]), _ptr(md["act_bytes"]), _ptr(md["ar_bytes"]),
                               _ptr(md["a2a_bytes"]), int(model["boundary_bytes"]),
                               int(bool(model.get("moe", False))), _ptr(prof), err)
        if not self._h:
            raise ValueError("oracle rejected inputs: " + err.value.decode())

    def price_plans(self, plans: dict) -> dict:
        """Multi-template plans (Algorithm 1): ``plans`` holds ``n_tmpl[n]``,
        ``S[t, n]``, ``M[t, n]`` and ``code[t, s, n]``.  Returns per template
        ``T``, ``bottleneck``, ``n_dp``, ``status`` ([t, n]) and per plan
        ``placed`` and ``thr`` (base micro-batches per second)."""
        nt = np.ascontiguousarray(plans["n_tmpl"], dtype=np.uint8)
        S = np.ascontiguousarray(plans["S"], dtype=np.uint8)
        M = np.ascontiguousarray(plans["M"], dtype=np.uint16)
        code = np.ascontiguousarray(plans["code"], dtype=np.uint8)
        tmax, n = S.shape
        s_max = int(code.shape[1])
        out = {"T": np.zeros((tmax, n), np.int64), "bottleneck": np.zeros((tmax, n), np.int64),
               "n_dp": np.zeros((tmax, n), np.uint16), "status": np.zeros((tmax, n), np.uint8),
               "placed": np.zeros(n, np.uint8), "thr": np.zeros(n, np.float64)}
        lib().orc_price_plans(self._h, n, tmax, _ptr(nt), _ptr(S), _ptr(M), _ptr(code), s_max, _ptr(out["T"]),
                              _ptr(out["bottleneck"]), _ptr(out["n_dp"]), _ptr(out["status"]),
                              _ptr(out["placed"]), _ptr(out["thr"]))
        return out

    def set_experts(self, expert_state=None, expert_param=None):
        """Expert tiling (§5.3): the expert parts of every layer's state and
        gradient bytes; ``None`` for both turns tiling off."""
        err = C.create_string_buffer(256)
        if expert_state is None and expert_param is None:
            rc = lib().orc_set_experts(self._h, None, None, err)
        else:
            es = np.ascontiguousarray(expert_state, dtype=np.int64)
            ep = np.ascontiguousarray(expert_param, dtype=np.int64)
            rc = lib().orc_set_experts(self._h, _ptr(es), _ptr(ep), err)
        if rc != 0:
            raise ValueError("oracle rejected expert bytes: " + err.value.decode())
        self.tiled = expert_state is not None
        return self

    def tiled_tables(self) -> dict:
        """Tiled prefix rows ``Pt[g, slot, l]`` (ns) and ``valid[g, slot]``."""
        Pt = np.zeros((self.n_types, 20, self.L + 1), np.int64)
        valid = np.zeros((self.n_types, 20), np.int32)
        lib().orc_tiled_tables(self._h, _ptr(Pt), _ptr(valid))
        return {"Pt": Pt, "valid": valid}

    def set_split(self, mode: str):
        """``"minmax"`` (PartitionLayers, the default) or ``"distribute"``
        (the paper's own proportional rule with its fixed alternatives)."""
        lib().orc_set_split(self._h, {"minmax": 0, "distribute": 1}[mode])
        return self

    def __del__(self):
        h = getattr(self, "_h", None)
        if h:
            lib().orc_destroy(h)
            self._h = None

    def tables(self) -> dict:
        """Quantised per-layer costs ``q[g, j, l]`` (ns), P2P constants
        ``p2p[g, h, same]`` (ns), largest node and slowest NIC per type."""
        q = np.zeros((self.n_types, 4, self.L), dtype=np.int64)
        p2p = np.zeros((8, 8, 2), dtype=np.int64)
        mx = np.zeros(self.n_types, dtype=np.int32)
        bw = np.zeros(self.n_types, dtype=np.int64)
        lib().orc_tables(self._h, _ptr(q), _ptr(p2p), _ptr(mx), _ptr(bw))
        return {"q": q, "P": np.concatenate([np.zeros((self.n_types, 4, 1), np.int64),
                                             np.cumsum(q, axis=2)], axis=2),
                "p2p": p2p, "maxnode": mx, "inter_bw": bw}

    def price(self, cands: dict, threads: int = 1, bounds: bool = True, tiling: bool = False) -> dict:
        """Price every candidate; returns T, bottleneck, n_dp, status, bounds[33, n]
        and, with ``tiling``, the chosen expert tiling of every stage
        ``tiling[32, n]`` (log2 EP | log2 ETP << 2)."""
        S = np.ascontiguousarray(cands["S"], dtype=np.uint8)
        M = np.ascontiguousarray(cands["M"], dtype=np.uint16)
        code = np.ascontiguousarray(cands["code"], dtype=np.uint8)
        n = int(S.shape[0])
        s_max = int(code.shape[0])
        out = {"T": np.zeros(n, np.int64), "bottleneck": np.zeros(n, np.int64),
               "n_dp": np.zeros(n, np.uint16), "status": np.zeros(n, np.uint8),
               "bounds": np.zeros((33, n), np.uint8) if bounds else None,
               "tiling": np.zeros((32, n), np.uint8) if tiling else None}
        used = lib().orc_price_tiled(self._h, n, _ptr(S), _ptr(M), _ptr(code), n, s_max,
                                     _ptr(out["T"]), _ptr(out["bottleneck"]), _ptr(out["n_dp"]),
                                     _ptr(out["status"]), _ptr(out["bounds"]), _ptr(out["tiling"]),
                                     int(threads))
        if used < 0:
            raise ValueError("expert tiling prices the min-max split only")
        out["threads"] = used
        return out


def topk(res: dict, M, k: int, base_index: int = 0) -> dict:
    """Top-``k`` OK candidates by throughput n*M/T (ties: smaller index)."""
    n = int(res["T"].shape[0])
    T = np.ascontiguousarray(res["T"], dtype=np.int64)
    nd = np.ascontiguousarray(res["n_dp"], dtype=np.uint16)
    st = np.ascontiguousarray(res["status"], dtype=np.uint8)
    Mm = np.ascontiguousarray(M, dtype=np.uint16)
    idx = np.zeros(k, np.int64)
    tt = np.zeros(k, np.int64)
    nm = np.zeros(k, np.uint32)
    cnt = lib().orc_topk(n, int(base_index), _ptr(T), _ptr(nd), _ptr(Mm), _ptr(st), int(k),
                         _ptr(idx), _ptr(tt), _ptr(nm))
    return {"count": cnt, "idx": idx[:cnt], "T": tt[:cnt], "nM": nm[:cnt]}


def partition_raw(P, c, W=None, cap=None):
    """Min-max contiguous partition on raw integer stage tables (test hook).

    ``P``: [S][L+1] int64 cost prefixes, ``c``: [S] per-stage constants,
    ``W``/``cap``: [S][L+1] memory prefixes and [S] capacities (default: no
    memory limit).  Returns ``(B*, bounds)`` or ``None`` when no split fits."""
    P = np.ascontiguousarray(P, dtype=np.int64)
    S, L1 = P.shape
    c = np.ascontiguousarray(c, dtype=np.int64)
    W = np.zeros_like(P) if W is None else np.ascontiguousarray(W, dtype=np.int64)
    cap = np.zeros(S, np.int64) if cap is None else np.ascontiguousarray(cap, dtype=np.int64)
    B = np.zeros(1, np.int64)
    a = np.zeros(S + 1, np.int32)
    ok = lib().orc_partition_raw(S, L1 - 1, _ptr(P), _ptr(c), _ptr(W), _ptr(cap), _ptr(B), _ptr(a))
    return (int(B[0]), a.tolist()) if ok else None


def replicas(node_gpus, group_gpus) -> int:
    """Largest replication count of ``group_gpus`` on ``node_gpus`` (one type)."""
    ng = np.ascontiguousarray(node_gpus, dtype=np.int32)
    gg = np.ascontiguousarray(group_gpus, dtype=np.int32)
    return int(lib().orc_replicas(len(ng), _ptr(ng), len(gg), _ptr(gg)))


# ------------------------------------------------------- micro-batch fill

def level_model(model: dict, level: int, profile_s=None) -> dict:
    """The model at micro-batch size 2**level times the base size (§5.3
    "Micro-batch size"): every quantity that grows with the tokens of a
    micro-batch -- FLOPs, stored activations, the TP all-reduce and EP
    all-to-all messages, the stage-boundary activation -- scales by
    2**level; parameter, gradient and optimizer-state bytes do not.
    ``profile_s`` (seconds per layer at this size, [types][4][L]) replaces
    the synthetic compute formula when given."""
    f = 1 << level
    out = dict(model)
    out["flops"] = np.asarray(model["flops"], np.float64) * float(f)
    for k in ("act_bytes", "ar_bytes", "a2a_bytes"):
        out[k] = np.asarray(model[k], np.int64) * f
    out["boundary_bytes"] = int(model["boundary_bytes"]) * f
    out["profile_s"] = None if profile_s is None else np.ascontiguousarray(profile_s, np.float64)
    return out


def price_mbs(cluster: dict, model: dict, cands: dict, levels: int, profiles=None, threads: int = 1,
              bounds: bool = True) -> dict:
    """Micro-batch-size fill (§5.3): price every candidate at micro-batch
    sizes 2**i times the base size, i = 0 .. levels-1, and keep the size
    with the shortest iteration time (ties: the smaller size).  A replica
    still processes M base micro-batches per iteration, so at size 2**i it
    runs M / 2**i micro-batches; a size that does not divide M is not
    priced for that candidate.  The size that fits nowhere makes no
    difference: a candidate that fits at no size keeps the base size's
    status.  Returns the fields of ``Oracle.price`` plus ``mbs`` (the chosen
    i; 0 for candidates that are not OK)."""
    M = np.asarray(cands["M"], dtype=np.int64)
    best = None
    for i in range(levels):
        prof = None if profiles is None else profiles[i]
        orc = Oracle(cluster, level_model(model, i, prof))
        div = (M % (1 << i)) == 0
        ci = dict(cands)
        ci["M"] = np.where(div, M >> i, 0).astype(np.uint16)  # M = 0 is INVALID
        r = orc.price(ci, threads=threads, bounds=bounds)
        if best is None:
            best = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in r.items()}
            best["mbs"] = np.zeros(len(M), np.uint8)
            continue
        take = (r["status"] == OK) & ((best["status"] != OK) | (r["T"] < best["T"]))
        for k in ("T", "bottleneck", "n_dp", "status"):
            best[k][take] = r[k][take]
        if bounds:
            best["bounds"][:, take] = r["bounds"][:, take]
        best["mbs"][take] = i
    return best
