"""Seeded synthetic workloads for batched candidate-plan pricing.

This module only *describes* inputs: GPU types, nodes, model layers and the
candidate pipeline structures (structural templates, paper §5.1).  It holds
none of the pricing arithmetic (no cost quantisation, partitioning, packing,
iteration time or ranking); both the CUDA library and the CPU oracle consume
the arrays it returns, so the two always see byte-identical inputs.

The paper's own workloads are profiled LLaMA/Qwen/MoE models on A100/H100/
A6000 clusters (§6) and a sweep of random plan structures on a 512-GPU
cluster (§3, "Pipeline structures" figure).  None of those profiles ship with
the paper, so every configuration here is a synthetic stand-in with the
shapes, sizes and value distributions listed in the workload recipe.

Units: time in seconds (float64) or FLOPs (float64), bytes and bytes/second as
int64, memory in decimal GB (1 GB = 1e9 B).

Candidate encoding (one byte per stage): bits 0-2 the GPU type index g,
bits 3-4 the log2 of the stage degree k (TP degree; EP degree for MoE models),
bits 5-7 zero.  Candidates are a structure of arrays: ``S`` (uint8 stage
count), ``M`` (uint16 microbatch count) and ``code`` (uint8, stage-major
planes: ``code[s, c]`` is stage ``s`` of candidate ``c``; planes at and beyond
a candidate's ``S`` are zero).
"""

from __future__ import annotations

import dataclasses
import itertools

import numpy as np

GB = 10**9
MAX_TYPES = 8
MAX_STAGES = 32
DEGREES = (1, 2, 4, 8)


@dataclasses.dataclass
class Workload:
    """One seeded problem instance: cluster, model and candidate batch."""

    name: str
    seed: int
    cluster: dict
    model: dict
    cands: dict
    meta: dict

    @property
    def n(self) -> int:
        return int(self.cands["S"].shape[0])


def encode(g, j):
    """Stage code byte for GPU type ``g`` and degree ``2**j``."""
    return (np.asarray(g, dtype=np.int64) | (np.asarray(j, dtype=np.int64) << 3)).astype(np.uint8)


def make_cluster(tflops, mem_bytes, intra_bw, nodes):
    """Cluster arrays from per-type properties and ``(type, gpus, nic_bw)`` nodes."""
    nodes = list(nodes)
    return {
        "tflops": np.asarray(tflops, dtype=np.float64),
        "mem_bytes": np.asarray(mem_bytes, dtype=np.int64),
        "intra_bw": np.asarray(intra_bw, dtype=np.int64),
        "node_type": np.asarray([t for t, _, _ in nodes], dtype=np.int32),
        "node_gpus": np.asarray([c for _, c, _ in nodes], dtype=np.int32),
        "node_nic": np.asarray([b for _, _, b in nodes], dtype=np.int64),
    }


def make_model(flops, param_bytes, state_bytes, act_bytes, ar_bytes, a2a_bytes,
               boundary_bytes, moe=False, profile_s=None, microbatch=1,
               expert_state=None, expert_param=None):
    """Model arrays (one entry per layer) plus model-wide scalars.  The
    optional expert parts of the state and gradient bytes (MoE expert
    blocks) feed the expert tiling."""
    L = len(flops)
    arr = lambda v, dt: np.broadcast_to(np.asarray(v, dtype=dt), (L,)).copy()
    return {
        "expert_state_bytes": None if expert_state is None else arr(expert_state, np.int64),
        "expert_param_bytes": None if expert_param is None else arr(expert_param, np.int64),
        "flops": arr(flops, np.float64),
        "param_bytes": arr(param_bytes, np.int64),
        "state_bytes": arr(state_bytes, np.int64),
        "act_bytes": arr(act_bytes, np.int64),
        "ar_bytes": arr(ar_bytes, np.int64),
        "a2a_bytes": arr(a2a_bytes, np.int64),
        "boundary_bytes": int(boundary_bytes),
        "moe": bool(moe),
        "microbatch": int(microbatch),
        "profile_s": None if profile_s is None else np.ascontiguousarray(profile_s, dtype=np.float64),
    }


def make_cands(S, M, code, s_max=None):
    """Candidate SoA; ``code`` is stage-major ``[s_max, n]``."""
    S = np.ascontiguousarray(S, dtype=np.uint8)
    M = np.ascontiguousarray(M, dtype=np.uint16)
    code = np.ascontiguousarray(code, dtype=np.uint8)
    if code.ndim == 1:
        code = code.reshape(-1, S.shape[0])
    if s_max is not None and code.shape[0] != s_max:
        raise ValueError("code planes do not match s_max")
    return {"S": S, "M": M, "code": code}


def from_structures(structs, M):
    """Candidates from a list of ``[(g, j), ...]`` stage lists (test helper)."""
    n = len(structs)
    s_max = max(1, max(len(s) for s in structs))
    code = np.zeros((s_max, n), dtype=np.uint8)
    S = np.zeros(n, dtype=np.uint8)
    for c, st in enumerate(structs):
        S[c] = len(st)
        for s, (g, j) in enumerate(st):
            code[s, c] = int(encode(g, j))
    Ms = np.broadcast_to(np.asarray(M, dtype=np.uint16), (n,)).copy()
    return make_cands(S, Ms, code)


# --------------------------------------------------------------------------
# transformer layer shapes (dense and MoE), bf16 mixed-precision Adam
# --------------------------------------------------------------------------

def _dense_layer(h, s, b, ffn=None):
    """FLOPs (fwd+bwd), parameter count and activation bytes of a dense block.

    ``ffn=None`` is the classic 4h MLP (12 h^2 parameters per block); an
    explicit ``ffn`` is a gated (SwiGLU) MLP with three h x ffn matrices.
    Activation bytes use 34*b*s*h (no s^2 term: fused attention).
    """
    params = 12 * h * h if ffn is None else 4 * h * h + 3 * h * ffn
    flops_fwd = 2 * b * s * params + 4 * b * s * s * h
    return 3.0 * flops_fwd, params, 34 * b * s * h


def _maxnode(cluster, g):
    m = cluster["node_gpus"][cluster["node_type"] == g]
    return int(m.max()) if m.size else 0


def _nodes_from_sizes(rng, n_types, total, sizes):
    """Node list whose sizes are drawn from ``sizes`` and sum to ``total``;
    every type owns at least one node."""
    sizes = sorted(sizes)
    out = []
    left = total
    while left > 0:
        fit = [z for z in sizes if z <= left]
        out.append(int(rng.choice(fit)))
        left -= out[-1]
    while len(out) < n_types:  # split the largest node until each type can own one
        i = int(np.argmax(out))
        if out[i] < 2:
            raise ValueError("too few GPUs for the number of types")
        half = out[i] // 2
        out[i] -= half
        out.append(half)
    types = list(range(n_types)) + [int(t) for t in rng.integers(0, n_types, len(out) - n_types)]
    rng.shuffle(types)
    return list(zip(types, out))


def _random_cands(rng, cluster, n, s_max, degree_set, M, moe=False, bad_frac=0.01, chunk=1 << 20):
    """Random structures: S ~ U{1..s_max}; per stage g ~ U(types), k ~ U over
    ``degree_set`` restricted to the largest node of g (the paper's TP mask,
    §5.1) unless ``moe`` (an EP degree may leave a node, §5.3).  About
    ``bad_frac`` of the candidates get one deliberately invalid stage.
    Generated in chunks of ``chunk`` candidates from one generator stream."""
    n_types = len(cluster["tflops"])
    tab = np.zeros((n_types, 4), dtype=np.uint8)
    cnt = np.zeros(n_types, dtype=np.uint32)
    big = np.full(n_types, 255, dtype=np.uint8)  # smallest j with 2**j above the largest node
    for t in range(n_types):
        mx = _maxnode(cluster, t)
        js = [int(np.log2(d)) for d in degree_set if moe or d <= mx]
        tab[t, : len(js)] = js
        cnt[t] = len(js)
        over = [jj for jj in range(4) if (1 << jj) > mx]
        if over:
            big[t] = over[0]
    S = np.empty(n, dtype=np.uint8)
    code = np.empty((s_max, n), dtype=np.uint8)
    live_rows = np.arange(s_max, dtype=np.uint8)[:, None]
    for lo in range(0, n, chunk):
        hi = min(n, lo + chunk)
        m = hi - lo
        Sc = rng.integers(1, s_max + 1, m, dtype=np.uint8)
        g = rng.integers(0, n_types, (s_max, m), dtype=np.uint8)
        r = rng.integers(0, 1 << 16, (s_max, m), dtype=np.uint32)
        u = (r * cnt[g]) >> 16
        j = tab[g, u]
        cc = (g | (j << 3)).astype(np.uint8)
        cc[live_rows >= Sc[None, :]] = 0
        S[lo:hi] = Sc
        code[:, lo:hi] = cc
    # deliberately invalid stages (~bad_frac): unknown type, reserved bits,
    # or (dense models) a degree above the largest node of the type
    n_bad = int(round(bad_frac * n))
    if n_bad:
        idx = np.sort(rng.choice(n, n_bad, replace=False))
        kinds = rng.integers(0, 3, n_bad)
        s = (rng.random(n_bad) * S[idx]).astype(np.int64)
        cur = code[s, idx].astype(np.int64)
        gc = cur & 7
        reserved = cur | 0x20
        unknown = np.full(n_bad, n_types, dtype=np.int64) if n_types < MAX_TYPES else reserved
        bj = big[gc].astype(np.int64)
        too_big = np.where(bj != 255, gc | (bj << 3), cur | 0x40)
        new = np.where(kinds == 0, unknown, np.where((kinds == 1) | moe, reserved, too_big))
        code[s, idx] = new.astype(np.uint8)
    if np.ndim(M) == 0:
        Ms = np.full(n, M, dtype=np.uint16)
    else:
        Ms = rng.choice(np.asarray(M, dtype=np.uint16), n)
    return make_cands(S, Ms, code)


# --------------------------------------------------------------------------
# the five workloads
# --------------------------------------------------------------------------

def tiny(seed=0, extended=False):
    """8-layer dense fp32 model on 4 GPUs of 2 types (speeds 1.0/0.5, 40/24 GB)
    in 2 nodes of 2; every structure with S <= 3 and TP in {1,2} (84), M = 8;
    ``extended`` repeats them for M in {1,2,4,8} (336)."""
    rng = np.random.default_rng(seed)
    cost_ms = rng.uniform(0.8, 1.2, 8)
    speed = [1.0, 0.5]
    tflops = [1000.0 * v for v in speed]
    flops = cost_ms * 1e-3 * 1000.0e12  # seconds at speed 1.0 times its FLOP/s
    cluster = make_cluster(tflops, [40 * GB, 24 * GB], [300 * GB, 300 * GB],
                           [(0, 2, 12_500_000_000), (1, 2, 12_500_000_000)])
    mb = 10**6
    model = make_model(flops, 50 * mb, 4 * 50 * mb, 20 * mb, 20 * mb, 0, 20 * mb)
    opts = [(g, j) for g in range(2) for j in range(2)]
    structs = [list(t) for S in (1, 2, 3) for t in itertools.product(opts, repeat=S)]
    Ms = (1, 2, 4, 8) if extended else (8,)
    all_structs = [st for _ in Ms for st in structs]
    M = np.repeat(np.asarray(Ms, dtype=np.uint16), len(structs))
    cands = from_structures(all_structs, M)
    meta = {"L": 8, "n_types": 2, "gpus": 4, "s_max": 3, "degrees": (1, 2), "topk": 16}
    return Workload("tiny_ext" if extended else "tiny", seed, cluster, model, cands, meta)


def _hetero_cluster(rng, n_types, total, node_sizes, speed_lo, mem_choices=None, mem_range=None):
    speeds = rng.uniform(speed_lo, 1.0, n_types)
    tflops = 1000.0 * speeds
    if mem_choices is not None:
        mem = rng.choice(np.asarray(mem_choices), n_types) * GB
    else:
        mem = rng.integers(mem_range[0], mem_range[1] + 1, n_types) * GB
    intra = rng.choice(np.asarray([64, 300, 900]), n_types) * GB
    nodes = _nodes_from_sizes(rng, n_types, total, node_sizes)
    nic = rng.choice(np.asarray([25, 100, 400]), len(nodes)) * (10**9 // 8)
    return make_cluster(tflops, mem, intra, [(t, c, int(b)) for (t, c), b in zip(nodes, nic)])


def _dense_model(L, h, s, b=1):
    flops, params, act = _dense_layer(h, s, b)
    pbytes = 2 * params  # bf16 weights; DP synchronises bf16 gradients
    return make_model(np.full(L, flops), pbytes, 16 * params, act, 2 * b * s * h, 0,
                      2 * b * s * h, microbatch=b)


def dense32(seed=0, n=100_000):
    """32-layer dense transformer (h 4096, seq 2048, b 1, bf16); 64 GPUs of 3
    types in nodes of 4/8; S <= 8, TP in {1,2,4}, M = 32."""
    rng = np.random.default_rng(seed)
    cluster = _hetero_cluster(rng, 3, 64, (4, 8), 0.3, mem_choices=(24, 40, 80))
    model = _dense_model(32, 4096, 2048)
    cands = _random_cands(rng, cluster, n, 8, (1, 2, 4), 32)
    meta = {"L": 32, "n_types": 3, "gpus": 64, "s_max": 8, "degrees": (1, 2, 4), "topk": 16}
    return Workload("dense32", seed, cluster, model, cands, meta)


def dense80(seed=0, n=1_000_000):
    """80-layer dense transformer (h 8192, seq 4096, bf16); 256 GPUs of 5 types
    in 4/8-GPU nodes; S <= 16, TP in {1,2,4,8}, M in {16,32,64,128}."""
    rng = np.random.default_rng(seed)
    cluster = _hetero_cluster(rng, 5, 256, (4, 8), 0.2, mem_choices=(16, 24, 40, 48, 80))
    model = _dense_model(80, 8192, 4096)
    cands = _random_cands(rng, cluster, n, 16, DEGREES, (16, 32, 64, 128))
    meta = {"L": 80, "n_types": 5, "gpus": 256, "s_max": 16, "degrees": DEGREES, "topk": 16}
    return Workload("dense80", seed, cluster, model, cands, meta)


def moe48(seed=0, n=1_000_000):
    """48-layer MoE model, dense and expert blocks alternating (64 experts,
    top-2, h 4096, ffn 14336, seq 2048, bf16); expert blocks carry an EP
    all-to-all of tokens x hidden x 2 B; 128 GPUs of 4 types in 4/8-GPU nodes;
    S <= 12, EP in {1,2,4,8}, M = 64."""
    rng = np.random.default_rng(seed)
    cluster = _hetero_cluster(rng, 4, 128, (4, 8), 0.3, mem_choices=(40, 80, 96, 141))
    h, ffn, s, b, E, top = 4096, 14336, 2048, 1, 64, 2
    d_flops, d_params, d_act = _dense_layer(h, s, b, ffn)
    e_params = 4 * h * h + E * 3 * h * ffn + h * E
    e_flops = 3.0 * (2 * b * s * (4 * h * h + top * 3 * h * ffn) + 4 * b * s * s * h)
    L = 48
    expert = np.arange(L) % 2 == 1
    params = np.where(expert, e_params, d_params)
    flops = np.where(expert, e_flops, d_flops)
    act = np.where(expert, 2 * d_act, d_act)
    tok = 2 * b * s * h
    ar = np.where(expert, tok // 2, tok)  # expert blocks: attention all-reduces only
    a2a = np.where(expert, tok, 0)
    e_only = np.where(expert, E * 3 * h * ffn, 0)  # the experts' own parameters
    model = make_model(flops, 2 * params, 16 * params, act, ar, a2a, tok, moe=True, microbatch=b,
                       expert_state=16 * e_only, expert_param=2 * e_only)
    cands = _random_cands(rng, cluster, n, 12, DEGREES, 64, moe=True)
    meta = {"L": L, "n_types": 4, "gpus": 128, "s_max": 12, "degrees": DEGREES, "topk": 16}
    return Workload("moe48", seed, cluster, model, cands, meta)


def moe16(seed=0, n=20_000):
    """16-layer MoE model for the expert-tiling tests: dense and expert
    blocks alternating (16 experts, top-2, h 2048, ffn 5632, seq 2048, bf16);
    64 GPUs of 3 types in 2/4/8-GPU nodes with 8-48 GB each, so that the
    expert state replicated by EDP fits on some stages and not on others;
    S <= 6, EP in {1,2,4,8}, M = 16."""
    rng = np.random.default_rng(seed)
    cluster = _hetero_cluster(rng, 3, 64, (2, 4, 8), 0.3, mem_range=(8, 48))
    h, ffn, s, b, E, top = 2048, 5632, 2048, 1, 16, 2
    d_flops, d_params, d_act = _dense_layer(h, s, b, ffn)
    e_only = E * 3 * h * ffn
    e_params = 4 * h * h + e_only + h * E
    e_flops = 3.0 * (2 * b * s * (4 * h * h + top * 3 * h * ffn) + 4 * b * s * s * h)
    L = 16
    expert = np.arange(L) % 2 == 1
    params = np.where(expert, e_params, d_params)
    tok = 2 * b * s * h
    model = make_model(np.where(expert, e_flops, d_flops), 2 * params, 16 * params,
                       np.where(expert, 2 * d_act, d_act), np.where(expert, tok // 2, tok),
                       np.where(expert, tok, 0), tok, moe=True, microbatch=b,
                       expert_state=np.where(expert, 16 * e_only, 0),
                       expert_param=np.where(expert, 2 * e_only, 0))
    cands = _random_cands(rng, cluster, n, 6, DEGREES, 16, moe=True)
    meta = {"L": L, "n_types": 3, "gpus": 64, "s_max": 6, "degrees": DEGREES, "topk": 16}
    return Workload("moe16", seed, cluster, model, cands, meta)


def stress128(seed=0, n=10_000_000):
    """128-layer dense model (h 12288, seq 4096, bf16); 1024 GPUs of 8 types
    in nodes of 2/4/8, speeds U[0.1,1], memory U[16,192] GB; S <= 32,
    TP in {1,2,4,8}, M = 256; streamed in batches of 1e6, global top-16."""
    rng = np.random.default_rng(seed)
    cluster = _hetero_cluster(rng, 8, 1024, (2, 4, 8), 0.1, mem_range=(16, 192))
    model = _dense_model(128, 12288, 4096)
    cands = _random_cands(rng, cluster, n, 32, DEGREES, 256)
    meta = {"L": 128, "n_types": 8, "gpus": 1024, "s_max": 32, "degrees": DEGREES,
            "topk": 16, "batch": 1_000_000}
    return Workload("stress128", seed, cluster, model, cands, meta)


CONFIGS = {
    "tiny": lambda seed=0, n=None: tiny(seed),
    "tiny_ext": lambda seed=0, n=None: tiny(seed, extended=True),
    "dense32": lambda seed=0, n=None: dense32(seed, 100_000 if n is None else n),
    "dense80": lambda seed=0, n=None: dense80(seed, 1_000_000 if n is None else n),
    "moe48": lambda seed=0, n=None: moe48(seed, 1_000_000 if n is None else n),
    "moe16": lambda seed=0, n=None: moe16(seed, 20_000 if n is None else n),
    "stress128": lambda seed=0, n=None: stress128(seed, 10_000_000 if n is None else n),
}


def mbs_profiles(w, levels: int, seed: int = 0):
    """Seeded per-size layer profiles for the micro-batch-size fill: a list
    of ``levels`` arrays [types][4][L] of seconds per layer at micro-batch
    2**i times the base size and TP degree 2**j.  The paper profiles every
    size on real GPUs (§5.3, "the profiled powers of two"); this stand-in
    draws per type a base time tau_g ~ U(0.5, 2) ms and a per-doubling
    efficiency rho_g ~ U(0.6, 0.95) (a larger micro-batch uses the GPU
    better), weights layer l by its share of the model's FLOPs, and sets
    t = tau_g * w_l * (1 + 0.15 j) / 2**j * (2 rho_g)**i."""
    rng = np.random.default_rng(0x5EED0 + seed)
    NT = int(w.cluster["tflops"].shape[0])
    fl = np.asarray(w.model["flops"], np.float64)
    wl = fl / fl.mean() if fl.mean() > 0 else np.ones_like(fl)
    tau = rng.uniform(0.5e-3, 2e-3, NT)
    rho = rng.uniform(0.6, 0.95, NT)
    j = np.arange(4, dtype=np.float64)
    out = []
    for i in range(levels):
        t = (tau[:, None, None] * (1.0 + 0.15 * j)[None, :, None] / (2.0 ** j)[None, :, None]
             * wl[None, None, :] * ((2.0 * rho) ** i)[:, None, None])
        out.append(np.ascontiguousarray(t))
    return out


def make_plans(w, n_plans: int, max_templates: int = 4, seed: int = 0) -> dict:
    """Seeded multi-template plans for ``w`` (same cluster and model): plan
    c holds n_tmpl[c] ~ U{1..max_templates} templates, each drawn from a pool
    of the workload's own candidate recipe (depth, GPU types and degrees,
    M).  Stage-major arrays per template slot: S[t, n], M[t, n],
    code[t, s, n]."""
    rng = np.random.default_rng(0xA11 + seed)
    pool = make_workload(w.name, seed=w.seed, n=n_plans * max_templates).cands
    pn = int(pool["S"].shape[0])
    pick = rng.integers(0, pn, (max_templates, n_plans))
    n_tmpl = rng.integers(1, max_templates + 1, n_plans).astype(np.uint8)
    return {"n_tmpl": n_tmpl, "S": pool["S"][pick], "M": pool["M"][pick],
            "code": np.ascontiguousarray(np.stack([pool["code"][:, pick[t]] for t in range(max_templates)]))}


def make_workload(name: str, seed: int = 0, n: int | None = None) -> Workload:
    """Build the named workload; ``n`` overrides the candidate count (same
    cluster, model and candidate distribution)."""
    return CONFIGS[name](seed, n)


def slice_cands(cands: dict, lo: int, hi: int) -> dict:
    """Candidates ``[lo, hi)`` as a new contiguous SoA."""
    return make_cands(cands["S"][lo:hi], cands["M"][lo:hi],
                      np.ascontiguousarray(cands["code"][:, lo:hi]))
