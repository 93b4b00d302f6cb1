"""Thin ctypes binding of ``libheddle.so`` (``include/heddle.h``).

Argument marshalling only: every function has the C name, packs Python /
numpy / torch arguments into the C structs and raises ``HeddleError`` on a
non-OK status.  All pricing runs in the library's CUDA kernels; there is no
fallback.  Device arrays are torch CUDA tensors (PyTorch supplies device
memory and streams); host arrays are numpy arrays or CPU tensors.
"""

from __future__ import annotations

import ctypes as C
import os

import numpy as np

# HEDDLE_LIB names another build of the library to load (the sanitizer and
# bounds-checked builds of the tests)
LIB_PATH = os.environ.get("HEDDLE_LIB") or os.path.join(os.path.dirname(os.path.abspath(__file__)), "libheddle.so")

MAX_TYPES, MAX_STAGES, MAX_LAYERS, MAX_TOPK = 8, 32, 255, 64
BOUND_PLANES = MAX_STAGES + 1
MODEL_MOE = 1
CAND_OK, CAND_OOM, CAND_NO_FIT, CAND_INVALID = 0, 1, 2, 3
STATUS_NAMES = {0: "OK", 1: "E_ARG", 2: "E_STATE", 3: "E_LIMIT", 4: "E_CUDA", 5: "E_NOMEM"}
E_ARG, E_STATE, E_LIMIT, E_CUDA, E_NOMEM = 1, 2, 3, 4, 5


class HeddleError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("%s: %s" % (STATUS_NAMES.get(status, status), msg))
        self.status = status


class heddle_gpu_type(C.Structure):
    _fields_ = [("tflops", C.c_double), ("mem_bytes", C.c_int64), ("intra_bw", C.c_int64)]


class heddle_node(C.Structure):
    _fields_ = [("type", C.c_int32), ("gpus", C.c_int32), ("nic_bw", C.c_int64)]


class heddle_layer(C.Structure):
    _fields_ = [("flops", C.c_double), ("param_bytes", C.c_int64), ("state_bytes", C.c_int64),
                ("act_bytes", C.c_int64), ("ar_bytes", C.c_int64), ("a2a_bytes", C.c_int64)]


class heddle_candidates(C.Structure):
    _fields_ = [("S", C.c_void_p), ("M", C.c_void_p), ("code", C.c_void_p), ("n", C.c_int64),
                ("plane_stride", C.c_int64), ("s_max", C.c_int32), ("reserved", C.c_int32),
                ("base_index", C.c_int64)]


class heddle_results(C.Structure):
    _fields_ = [("T", C.c_void_p), ("bottleneck", C.c_void_p), ("n_dp", C.c_void_p),
                ("status", C.c_void_p), ("bounds", C.c_void_p)]


MAX_TEMPLATES = 4
CAND_SKIPPED = 4


class heddle_plans(C.Structure):
    _fields_ = [("n", C.c_int64), ("slots", C.c_int32), ("reserved", C.c_int32),
                ("n_templates", C.c_void_p), ("t", heddle_candidates * MAX_TEMPLATES)]


class heddle_plan_results(C.Structure):
    _fields_ = [("t", heddle_results * MAX_TEMPLATES), ("placed", C.c_void_p), ("thr", C.c_void_p)]


class heddle_topk_state(C.Structure):
    _fields_ = [("k", C.c_int32), ("count", C.c_int32), ("idx", C.c_int64 * MAX_TOPK),
                ("T", C.c_int64 * MAX_TOPK), ("nM", C.c_uint32 * MAX_TOPK)]


TOPK_STATE_BYTES = C.sizeof(heddle_topk_state)

EXPORTS = ["heddle_create", "heddle_destroy", "heddle_last_error", "heddle_load_cluster",
           "heddle_load_model", "heddle_price_candidates", "heddle_topk_reset", "heddle_topk",
           "heddle_price_topk_host", "heddle_get_tables", "heddle_device_errors",
           "heddle_count_next", "heddle_work_counters", "heddle_set_search", "heddle_get_search", "heddle_set_thread_search_min",
           "heddle_price_topk", "heddle_topk_noalloc", "heddle_time_phases", "heddle_phase_times",
           "heddle_load_mbs", "heddle_price_mbs", "heddle_price_plans", "heddle_load_experts",
           "heddle_price_tiled", "heddle_set_chunk"]
MAX_MBS_LEVELS = 4
PHASES = ("screen", "search", "topk")
TOPK_NOALLOC_MAX_N = 4194304
SEARCH_AUTO, SEARCH_GENERAL, SEARCH_EQUAL_LAYERS, SEARCH_DISTRIBUTE, SEARCH_TILED = 0, 1, 2, 3, 4

_lib = None


def load_library(path: str = LIB_PATH):
    """Load ``libheddle.so``; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError("libheddle.so is not built (%s); run __graft_entry__.build()" % path)
    L = C.CDLL(path)
    p, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
    sig = {
        "heddle_create": (i32, [C.POINTER(C.c_void_p), i32]),
        "heddle_destroy": (None, [p]),
        "heddle_last_error": (C.c_char_p, [p]),
        "heddle_load_cluster": (i32, [p, p, i32, p, i32]),
        "heddle_load_model": (i32, [p, p, i32, i64, i32, p]),
        "heddle_price_candidates": (i32, [p, p, p, p]),
        "heddle_topk_reset": (i32, [p, p, i32, p]),
        "heddle_topk": (i32, [p, p, p, p, p]),
        "heddle_price_topk": (i32, [p, p, p, p, p]),
        "heddle_topk_noalloc": (i32, [p, p, p, p]),
        "heddle_price_topk_host": (i32, [p, p, p, p, i64, p]),
        "heddle_get_tables": (i32, [p, p, p]),
        "heddle_device_errors": (i32, [p, C.POINTER(C.c_uint32)]),
        "heddle_count_next": (i32, [p, i32]),
        "heddle_work_counters": (i32, [p, C.POINTER(C.c_uint64)]),
        "heddle_set_search": (i32, [p, i32]),
        "heddle_set_thread_search_min": (i32, [p, i32]),
        "heddle_get_search": (i32, [p, C.POINTER(C.c_int32)]),
        "heddle_time_phases": (i32, [p, i32]),
        "heddle_load_mbs": (i32, [p, i32, p]),
        "heddle_price_plans": (i32, [p, p, p, p]),
        "heddle_price_mbs": (i32, [p, p, p, p, p]),
        "heddle_load_experts": (i32, [p, p, p, i32]),
        "heddle_price_tiled": (i32, [p, p, p, p, p]),
        "heddle_set_chunk": (i32, [p, i64]),
        "heddle_phase_times": (i32, [p, C.POINTER(C.c_double), C.POINTER(C.c_int64)]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def _check(ctx, status):
    if status != 0:
        msg = load_library().heddle_last_error(ctx)
        raise HeddleError(status, (msg or b"").decode())


def _ptr(a):
    """Address of a torch tensor or numpy array (None -> NULL)."""
    if a is None:
        return None
    if hasattr(a, "data_ptr"):
        return a.data_ptr()
    return a.ctypes.data


def _stream(stream):
    if stream is None:
        try:
            import torch
            return torch.cuda.current_stream().cuda_stream
        except Exception:
            return None
    return getattr(stream, "cuda_stream", stream)


# ------------------------------------------------------------------ calls

def heddle_create(device: int = 0):
    h = C.c_void_p()
    st = load_library().heddle_create(C.byref(h), int(device))
    if st != 0:
        raise HeddleError(st, "heddle_create(device=%d) failed" % device)
    return h


def heddle_destroy(ctx):
    if ctx:
        load_library().heddle_destroy(ctx)


def heddle_last_error(ctx) -> str:
    return (load_library().heddle_last_error(ctx) or b"").decode()


def heddle_load_cluster(ctx, cluster: dict):
    nt = len(cluster["tflops"])
    types = (heddle_gpu_type * nt)(*[heddle_gpu_type(float(cluster["tflops"][g]),
                                                     int(cluster["mem_bytes"][g]),
                                                     int(cluster["intra_bw"][g])) for g in range(nt)])
    nn = len(cluster["node_type"])
    nodes = (heddle_node * nn)(*[heddle_node(int(cluster["node_type"][b]), int(cluster["node_gpus"][b]),
                                             int(cluster["node_nic"][b])) for b in range(nn)])
    _check(ctx, load_library().heddle_load_cluster(ctx, types, nt, nodes, nn))


def heddle_load_model(ctx, model: dict):
    L = len(model["flops"])
    layers = (heddle_layer * L)(*[heddle_layer(float(model["flops"][l]), int(model["param_bytes"][l]),
                                               int(model["state_bytes"][l]), int(model["act_bytes"][l]),
                                               int(model["ar_bytes"][l]), int(model["a2a_bytes"][l]))
                                  for l in range(L)])
    prof = model.get("profile_s")
    if prof is not None:
        prof = np.ascontiguousarray(prof, dtype=np.float64)
    flags = MODEL_MOE if model.get("moe") else 0
    _check(ctx, load_library().heddle_load_model(ctx, layers, L, int(model["boundary_bytes"]), flags,
                                                 None if prof is None else prof.ctypes.data))


def make_candidates(cands: dict, lo: int = 0, hi: int | None = None, base_index: int = 0):
    """C struct for candidates ``[lo, hi)`` of a stage-major SoA (device or host)."""
    n_all = int(cands["S"].shape[0])
    hi = n_all if hi is None else hi
    code = cands["code"]
    itemsize = 1
    return heddle_candidates(_ptr(cands["S"]) + lo if hi > lo else _ptr(cands["S"]),
                             _ptr(cands["M"]) + 2 * lo if hi > lo else _ptr(cands["M"]),
                             _ptr(code) + itemsize * lo if hi > lo else _ptr(code),
                             hi - lo, n_all, int(code.shape[0]), 0, base_index + lo)


def make_results(res: dict, lo: int = 0, hi: int | None = None):
    """C struct for results ``[lo, hi)`` (bounds must span exactly the batch)."""
    n = int(res["T"].shape[0])
    hi = n if hi is None else hi
    b = res.get("bounds")
    return heddle_results(_ptr(res["T"]) + 8 * lo, _ptr(res["bottleneck"]) + 8 * lo,
                          _ptr(res["n_dp"]) + 2 * lo, _ptr(res["status"]) + lo,
                          None if b is None else _ptr(b))


def heddle_price_candidates(ctx, cands, results, stream=None):
    """Price device candidates (``heddle_candidates`` struct or SoA dict of
    CUDA tensors) into device results (struct or dict of CUDA tensors)."""
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    _check(ctx, load_library().heddle_price_candidates(ctx, C.byref(c), C.byref(r), _stream(stream)))


def heddle_load_mbs(ctx, levels: int, profiles=None):
    """Prepare the micro-batch-size fill for sizes 2**i, i < ``levels``;
    ``profiles``: optional per-size seconds per layer, a sequence of
    ``levels`` arrays [types][4][L] (host)."""
    prof = None
    if profiles is not None:
        prof = np.ascontiguousarray(np.stack([np.asarray(x, np.float64) for x in profiles]), dtype=np.float64)
    _check(ctx, load_library().heddle_load_mbs(ctx, int(levels), None if prof is None else prof.ctypes.data))


def heddle_price_mbs(ctx, cands, results, mbs=None, stream=None):
    """Price device candidates at every loaded micro-batch size and keep the
    fastest per candidate; ``mbs`` (optional device uint8 tensor) receives
    the chosen size's log2."""
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    _check(ctx, load_library().heddle_price_mbs(ctx, C.byref(c), C.byref(r),
                                                None if mbs is None else _ptr(mbs), _stream(stream)))


def heddle_set_chunk(ctx, chunk: int):
    """Chunk size of the pricing calls (1 .. 2**20); a call of several
    chunks pipelines them over two work streams."""
    _check(ctx, load_library().heddle_set_chunk(ctx, int(chunk)))


def heddle_load_experts(ctx, expert_state=None, expert_param=None):
    """Expert tiling (§5.3): the experts' part of every layer's state and
    gradient bytes (host arrays); ``None`` for both turns tiling off."""
    if expert_state is None and expert_param is None:
        _check(ctx, load_library().heddle_load_experts(ctx, None, None, 0))
        return
    es = np.ascontiguousarray(expert_state, dtype=np.int64)
    ep = np.ascontiguousarray(expert_param, dtype=np.int64)
    if es.shape != ep.shape or es.ndim != 1:
        raise ValueError("expert_state and expert_param must be 1-D arrays of one length")
    _check(ctx, load_library().heddle_load_experts(ctx, es.ctypes.data, ep.ctypes.data, int(es.shape[0])))


def heddle_price_tiled(ctx, cands, results, tiling=None, stream=None):
    """Price device candidates with expert tiling; ``tiling`` (optional
    device uint8 tensor [32, n]) receives each stage's log2 EP | log2 ETP << 2."""
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    _check(ctx, load_library().heddle_price_tiled(ctx, C.byref(c), C.byref(r),
                                                  None if tiling is None else _ptr(tiling), _stream(stream)))


def plans_to_device(plans: dict, device="cuda") -> dict:
    """Copy host plan arrays (n_tmpl[n], S[t, n], M[t, n], code[t, s, n]) to
    CUDA tensors, one candidate SoA per template slot."""
    import torch
    slots = [cands_to_device({"S": plans["S"][t], "M": plans["M"][t], "code": plans["code"][t]}, device)
             for t in range(plans["S"].shape[0])]
    return {"n_tmpl": torch.from_numpy(np.ascontiguousarray(plans["n_tmpl"])).to(device), "slots": slots}


def alloc_plan_results(n: int, slots: int, bounds: bool = False, device="cuda") -> dict:
    import torch
    return {"slots": [alloc_results(n, bounds=bounds, device=device) for _ in range(slots)],
            "placed": torch.empty(n, dtype=torch.uint8, device=device),
            "thr": torch.empty(n, dtype=torch.float64, device=device)}


def heddle_price_plans(ctx, dplans: dict, pres: dict, stream=None):
    """Price device plans (``plans_to_device``) into ``alloc_plan_results``."""
    slots = len(dplans["slots"])
    n = int(dplans["n_tmpl"].shape[0])
    pl = heddle_plans()
    pl.n = n
    pl.slots = slots
    pl.n_templates = _ptr(dplans["n_tmpl"])
    pr = heddle_plan_results()
    for t in range(slots):
        pl.t[t] = make_candidates(dplans["slots"][t])
        pr.t[t] = make_results(pres["slots"][t])
    pr.placed = _ptr(pres["placed"])
    pr.thr = _ptr(pres["thr"])
    _check(ctx, load_library().heddle_price_plans(ctx, C.byref(pl), C.byref(pr), _stream(stream)))


def heddle_topk_reset(ctx, state, k: int, stream=None):
    _check(ctx, load_library().heddle_topk_reset(ctx, _ptr(state), int(k), _stream(stream)))


def heddle_topk(ctx, cands, results, state, stream=None):
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    _check(ctx, load_library().heddle_topk(ctx, C.byref(c), C.byref(r), _ptr(state), _stream(stream)))


def heddle_price_topk(ctx, cands, results, state, stream=None):
    """Price device candidates and merge their OK ones into the device state."""
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    _check(ctx, load_library().heddle_price_topk(ctx, C.byref(c), C.byref(r), _ptr(state), _stream(stream)))


def heddle_topk_noalloc(cands, results, state, stream=None):
    """Allocation-free top-k merge (no context; current device); see the header."""
    c = cands if isinstance(cands, heddle_candidates) else make_candidates(cands)
    r = results if isinstance(results, heddle_results) else make_results(results)
    st = load_library().heddle_topk_noalloc(C.byref(c), C.byref(r), _ptr(state), _stream(stream))
    if st != 0:
        raise HeddleError(st, "heddle_topk_noalloc failed")


def heddle_price_topk_host(ctx, cands: dict, results: dict | None, state: heddle_topk_state,
                           batch: int, stream=None):
    """Host-buffer path: host SoA in, host results (optional) and host state out."""
    c = make_candidates(cands)
    r = heddle_results() if results is None else heddle_results(
        _ptr(results.get("T")), _ptr(results.get("bottleneck")), _ptr(results.get("n_dp")),
        _ptr(results.get("status")), _ptr(results.get("bounds")))
    _check(ctx, load_library().heddle_price_topk_host(ctx, C.byref(c), C.byref(r), C.byref(state),
                                                      int(batch), _stream(stream)))


def heddle_get_tables(ctx, n_types: int, n_layers: int):
    q = np.zeros((n_types, 4, n_layers), np.int64)
    p2p = np.zeros((8, 8, 2), np.int64)
    _check(ctx, load_library().heddle_get_tables(ctx, q.ctypes.data, p2p.ctypes.data))
    return q, p2p


def heddle_device_errors(ctx) -> int:
    f = C.c_uint32(0)
    _check(ctx, load_library().heddle_device_errors(ctx, C.byref(f)))
    return int(f.value)


def heddle_count_next(ctx, enable: bool = True):
    _check(ctx, load_library().heddle_count_next(ctx, int(bool(enable))))


def heddle_work_counters(ctx):
    out = (C.c_uint64 * 3)()
    _check(ctx, load_library().heddle_work_counters(ctx, out))
    return {"checks": int(out[0]), "probes": int(out[1]), "priced": int(out[2])}


def heddle_time_phases(ctx, enable: bool = True):
    _check(ctx, load_library().heddle_time_phases(ctx, int(bool(enable))))


def heddle_phase_times(ctx):
    """Summed device milliseconds and kernel launches per pricing phase
    since the last read: {"screen": (ms, launches), "search": ..., "topk": ...}."""
    ms = (C.c_double * len(PHASES))()
    n = (C.c_int64 * len(PHASES))()
    _check(ctx, load_library().heddle_phase_times(ctx, ms, n))
    return {name: (float(ms[i]), int(n[i])) for i, name in enumerate(PHASES)}


def heddle_set_search(ctx, mode: int):
    _check(ctx, load_library().heddle_set_search(ctx, int(mode)))


def heddle_set_thread_search_min(ctx, min_entries: int):
    """Bucketed entries from which the general search runs its
    thread-per-entry kernel (< 0: the default, 32 x the SM count)."""
    _check(ctx, load_library().heddle_set_thread_search_min(ctx, int(min_entries)))


def heddle_get_search(ctx) -> int:
    m = C.c_int32(0)
    _check(ctx, load_library().heddle_get_search(ctx, C.byref(m)))
    return int(m.value)


# ------------------------------------------------------------- marshalling helpers

def topk_state_from_bytes(buf) -> dict:
    """Decode a ``heddle_topk_state`` from raw bytes (numpy uint8 / CPU tensor)."""
    raw = bytes(np.asarray(buf, dtype=np.uint8).tobytes())
    s = heddle_topk_state.from_buffer_copy(raw[:TOPK_STATE_BYTES])
    return topk_state_to_dict(s)


def topk_state_to_dict(s: heddle_topk_state) -> dict:
    cnt = int(s.count)
    return {"k": int(s.k), "count": cnt, "idx": np.array(s.idx[:cnt], np.int64),
            "T": np.array(s.T[:cnt], np.int64), "nM": np.array(s.nM[:cnt], np.uint32)}


def new_topk_state(k: int) -> heddle_topk_state:
    s = heddle_topk_state()
    s.k = k
    s.count = 0
    return s


# ------------------------------------------------------- torch device helpers

def cands_to_device(cands: dict, device="cuda") -> dict:
    """Copy a host SoA to CUDA tensors (uint16 travels as its int16 bit pattern)."""
    import torch
    return {"S": torch.from_numpy(np.ascontiguousarray(cands["S"])).to(device),
            "M": torch.from_numpy(np.ascontiguousarray(cands["M"]).view(np.int16)).to(device),
            "code": torch.from_numpy(np.ascontiguousarray(cands["code"])).to(device)}


def alloc_results(n: int, bounds: bool = False, device="cuda") -> dict:
    import torch
    return {"T": torch.empty(n, dtype=torch.int64, device=device),
            "bottleneck": torch.empty(n, dtype=torch.int64, device=device),
            "n_dp": torch.empty(n, dtype=torch.int16, device=device),
            "status": torch.empty(n, dtype=torch.uint8, device=device),
            "bounds": torch.empty((BOUND_PLANES, n), dtype=torch.uint8, device=device) if bounds else None}


def results_to_numpy(res: dict) -> dict:
    out = {"T": res["T"].cpu().numpy(), "bottleneck": res["bottleneck"].cpu().numpy(),
           "n_dp": res["n_dp"].cpu().numpy().view(np.uint16), "status": res["status"].cpu().numpy()}
    out["bounds"] = None if res.get("bounds") is None else res["bounds"].cpu().numpy()
    return out


def alloc_topk_state(device="cuda"):
    import torch
    return torch.zeros(TOPK_STATE_BYTES, dtype=torch.uint8, device=device)


def read_topk_state(state) -> dict:
    return topk_state_from_bytes(state.cpu().numpy())
