"""Benchmark: candidate plans priced per second on one GB300.

A step prices the whole 128-layer stress workload -- 1e7 candidate pipeline
structures for a 1024-GPU cluster of 8 types (S <= 32, TP in {1,2,4,8},
M = 256) -- as ten device-resident batches of 1e6 (PartitionLayers +
Evaluate kernel, then the block/grid top-k merge into one top-16 state).
Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference]

N > 1 runs under torchrun, one rank per GPU; every rank prices its own 1e7
candidates (weak scaling) and the per-rank top-16 lists are merged on the
host.  ``--impl reference`` times the CPU oracle on the host cores instead.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "candidate plans priced/sec on 1 GB300 (and % of ALU/HBM roofline)"
UNIT = "candidates/s"
WORKLOAD = "stress128"
WORKLOAD_DESC = ("stress128: 128-layer dense model (h 12288, seq 4096, bf16), 1024 GPUs of 8 types in "
                 "nodes of 2/4/8, 1e7 candidates per step in one call, priced in 10 chunks of 1e6 pipelined over four "
                 "work streams, S<=32, "
                 "TP in {1,2,4,8}, M=256, global top-16")
# Algorithmic integer work per counted unit, in 32-bit lane operations.
# General search, unit = one interval check (as the warp-per-entry kernel
# performs them: whole 32-position words per round, so it counts the
# positions a serial probe would skip as well): stage cost P[j]-P[i]+c against
# B (int64 subtract, add, compare) and stage memory (S[j]-S[i]) +
# f*(A[j]-A[i]) against the capacity (two int64 subtracts, one multiply by a
# 32-bit count, one add, one compare): 8 int64 ops = 16.
# Equal-layer search, unit = one stage of a searched candidate, counted once
# whatever the number of probes: the work of checking B* and evaluating the
# plan.  One exact stage capacity min(m, floor((B-c)/q)) at B*: B-c (2),
# x >= m*q (multiply 2, compare 2), the quotient estimate and its two
# multiply-compare corrections (10), the running sum (1), the snapping
# values c + k*q (4) and c + (k+1)*q (4) with their max / min (4): 29.
# Evaluate: stage time (a_{s+1}-a_s)*q + c (4), its max and sum (4), the
# boundary max(a_s + 1, L - suffix) with the running count (4), the
# stage's gradient bytes (2) and bandwidth (2), the exact ratio comparison
# of two 64x64->128-bit products (20): 36.  Together 65.
OPS_PER_UNIT = {1: 16, 2: 65}
# Screen (decode, validate, DP degree, memory screen), per candidate, in
# 32-bit lane operations: the depth and M checks (2) and the status decision
# (3); per stage the admissibility bit (1), its units added to its type's
# demand word (2), the in-flight count min(S - s, M) (2), the run-table row
# offset (1) and the running sum and minimum of the runs (2): 8; per type
# used, its demand fields unpacked (2), and per (type, degree) used the
# cumulative demand (1), the quotient capacity / demand as a multiply-high
# and shift (2) and the running minimum (1): 4.  Top-k, per searched
# candidate: its throughput key and the threshold comparison (4).
SCREEN_OPS = {"candidate": 5, "stage": 8, "type": 2, "pair": 4}
TOPK_OPS_PER_SEARCHED = 4


def screen_ops(cands) -> int:
    """Algorithmic lane operations of the screen over a candidate set."""
    S = cands["S"].astype(np.int64)
    code = cands["code"]
    pairs = np.zeros(S.shape[0], np.uint64)
    types = np.zeros(S.shape[0], np.uint32)
    for s_ in range(code.shape[0]):
        live = S > s_
        b = code[s_].astype(np.uint64) & 31
        pairs |= np.where(live, np.uint64(1) << b, np.uint64(0))
        types |= np.where(live, np.uint32(1) << (code[s_].astype(np.uint32) & 7), np.uint32(0))
    npairs = sum(int(((pairs >> np.uint64(i)) & np.uint64(1)).sum()) for i in range(32))
    ntypes = sum(int(((types >> np.uint32(i)) & np.uint32(1)).sum()) for i in range(8))
    return (SCREEN_OPS["candidate"] * S.shape[0] + SCREEN_OPS["stage"] * int(S.sum()) +
            SCREEN_OPS["type"] * ntypes + SCREEN_OPS["pair"] * npairs)


SEARCH_NAMES = {1: "general interval search", 2: "equal-layer closed form"}
SEARCH_KERNELS = {1: "gsearch_kernel + wsearch_kernel (general threshold search: one thread per single-fit "
                     "entry when there are at least 32 per SM, one warp per entry for the rest)",
                  2: "eq_search_kernel (equal-layer closed form)"}
LANES_PER_SM = 128  # 4 SM sub-partitions x 32 lanes issue per clock; the SM count comes from the device

# DRAM bytes (read + write) of one search launch on a 1e6-candidate batch of
# the stress workload, from an ncu capture, with the SHA-256 of the kernel
# sources it was taken on; reported as null once those sources change.
TRAFFIC = {2: {"bytes": 15419136, "batch": 1000000,
              "sha256": "fa830009fc0782dd6d8b53c00ed919aa761afde74f5a55b872bdc130ccdc3819"}}
TRAFFIC_SOURCES = {1: ["heddle_gsearch.cu", "heddle_wsearch.cu", "heddle_wprobe.cuh", "heddle_internal.cuh"],
                   2: ["heddle_eqsearch.cu", "heddle_internal.cuh"]}


def traffic_per_launch(search, batch):
    import hashlib
    rec = TRAFFIC.get(search)
    if rec is None or batch != rec["batch"]:
        return None
    hs = hashlib.sha256()
    for f in TRAFFIC_SOURCES[search]:
        with open(os.path.join(ROOT, "paper_2609_34244_gb300", "csrc", f), "rb") as fh:
            hs.update(fh.read())
    return rec["bytes"] if hs.hexdigest() == rec["sha256"] else None


def gpu_numa(dev):
    """NUMA node and local CPUs of the GPU from sysfs (empty when unknown)."""
    import torch
    p = torch.cuda.get_device_properties(dev)
    try:
        bus = "%04x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
    except AttributeError:
        return {}
    out = {"pci": bus}
    base = "/sys/bus/pci/devices/" + bus
    try:
        with open(base + "/numa_node") as f:
            out["gpu_numa_node"] = int(f.read().strip())
    except (OSError, ValueError):
        pass
    try:
        with open(base + "/local_cpulist") as f:
            txt = f.read().strip()
        cpus = set()
        for part in txt.split(","):
            if "-" in part:
                a, b = part.split("-")
                cpus.update(range(int(a), int(b) + 1))
            elif part:
                cpus.add(int(part))
        out["local_cpulist"] = txt
        out["cpus"] = sorted(cpus)
    except (OSError, ValueError):
        pass
    return out


def h2d_copy_gbs(nbytes):
    """Host-to-device copy rate from pinned memory, GB/s (best of 5)."""
    import torch
    src = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    src.numpy()[...] = 1
    dst = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    dst.copy_(src, non_blocking=True)
    torch.cuda.synchronize()
    best = None
    for _ in range(5):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        dst.copy_(src, non_blocking=True)
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
        best = ms if best is None else min(best, ms)
    del src, dst
    return nbytes / (best / 1e3) / 1e9


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": 6800.0, "sm_max_mhz": 2070.0}, "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="clocks", suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def oracle_rate(w, seconds, threads, max_n=None):
    """Oracle candidates/s on a bounded sample sized for about ``seconds``."""
    from oracle import oracle as O
    from paper_2609_34244_gb300 import workloads as W
    orc = O.Oracle(w.cluster, w.model)
    probe_n = min(w.n, 4 * threads * 8)
    sub = W.slice_cands(w.cands, 0, probe_n)
    t0 = time.perf_counter()
    orc.price(sub, threads=threads, bounds=False)
    dt = max(time.perf_counter() - t0, 1e-6)
    n = int(min(w.n, max(probe_n, probe_n * seconds / dt)))
    if max_n:
        n = min(n, max_n)
    sub = W.slice_cands(w.cands, 0, n)
    t0 = time.perf_counter()
    used = orc.price(sub, threads=threads, bounds=False)["threads"]
    dt = time.perf_counter() - t0
    return n / dt, n, used, dt


def run_reference(args, w):
    """The CPU oracle as the reference arm: each step prices a bounded sample."""
    threads = os.cpu_count() or 1
    _, n, used, _ = oracle_rate(w, 4.0, threads)
    from oracle import oracle as O
    from paper_2609_34244_gb300 import workloads as W
    orc = O.Oracle(w.cluster, w.model)
    sub = W.slice_cands(w.cands, 0, n)
    for _ in range(args.warmup):
        orc.price(sub, threads=threads, bounds=False)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        orc.price(sub, threads=threads, bounds=False)
    dt = time.perf_counter() - t0
    value = n * args.steps / dt
    sample = "first %d candidates of %s seed 0 per step, %d host threads" % (n, WORKLOAD, used)
    # n_gpus: the N of the run this arm is paired with (the oracle itself
    # runs on rank 0's host cores; `cpu_baseline.cores` says how many)
    return {"metric": METRIC, "value": value, "unit": UNIT, "impl": "reference", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
            "data": "synthetic",
            "config": {"workload": WORKLOAD_DESC, "candidates_per_step": n, "sample": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": used, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# The five workloads of the benchmark suite, each measured on its own in
# the default run (the headline line stays stress128).
PER_CONFIG = ("tiny", "dense32", "dense80", "moe48", "stress128")


def measure_config(h, name, peaks, sms, steps=20, cpu_seconds=3.0, main=None):
    """Candidates/s, per-candidate and single-batch latency, the dominant
    kernel's own launch time and roofline fraction, and the oracle's rate on
    the host cores in the same run, for one workload at its defining size
    (one pricing call over all candidates, chunks of 1e6).  Inputs smaller
    than L2 are preceded by an L2 flush outside each timed step."""
    import torch
    from paper_2609_34244_gb300 import workloads as W
    w = W.make_workload(name, seed=0)
    n = w.n
    batch = min(1_000_000, n)
    stream = torch.cuda.current_stream()
    ctx = h.heddle_create(torch.cuda.current_device())
    try:
        h.heddle_load_cluster(ctx, w.cluster)
        h.heddle_load_model(ctx, w.model)
        h.heddle_set_chunk(ctx, batch)
        search = h.heddle_get_search(ctx)
        dc = h.cands_to_device(w.cands)
        res = h.alloc_results(n)
        state = h.alloc_topk_state()
        bat = [(h.make_candidates(dc, lo, min(n, lo + batch)), h.make_results(res, lo, min(n, lo + batch)))
               for lo in range(0, n, batch)]
        for c, r in bat:
            h.heddle_count_next(ctx, True)
            h.heddle_price_candidates(ctx, c, r, stream)
        work = h.heddle_work_counters(ctx)
        allc, allr = h.make_candidates(dc), h.make_results(res)
        in_bytes = sum(int(v.numel() * v.element_size()) for v in dc.values())
        flush = torch.empty(256 << 20, dtype=torch.uint8, device="cuda") if in_bytes < (200 << 20) else None

        def step():
            h.heddle_topk_reset(ctx, state, 16, stream)
            h.heddle_price_topk(ctx, allc, allr, state, stream)

        for _ in range(3):
            step()
        torch.cuda.synchronize()
        evs = []
        for _ in range(steps):
            if flush is not None:
                flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step()
            e1.record(stream)
            evs.append((e0, e1))
        torch.cuda.synchronize()
        per = [a.elapsed_time(b) for a, b in evs]
        ms = float(np.mean(per))
        lat = []
        c0, r0 = bat[0]
        for _ in range(10):
            t0 = time.perf_counter()
            h.heddle_topk_reset(ctx, state, 16, stream)
            h.heddle_price_topk(ctx, c0, r0, state, stream)
            torch.cuda.synchronize()
            lat.append((time.perf_counter() - t0) * 1e3)
        # the search kernel's own launches: one call per batch, no overlap
        h.heddle_time_phases(ctx, True)
        for _ in range(3):
            h.heddle_topk_reset(ctx, state, 16, stream)
            for c, r in bat:
                h.heddle_price_topk(ctx, c, r, state, stream)
        torch.cuda.synchronize()
        h.heddle_time_phases(ctx, False)
        ph = h.heddle_phase_times(ctx)
        errors = h.heddle_device_errors(ctx)
    finally:
        h.heddle_destroy(ctx)
    peak = sms * LANES_PER_SM * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    s_ms, s_launches = ph["search"]
    chunks = max(1, ph["screen"][1])
    ops = work["checks"] * OPS_PER_UNIT.get(search, 0)
    tops = ops * 3 / (s_ms / 1e3) / 1e12 if s_ms > 0 else None
    threads = os.cpu_count() or 1
    rate, ncpu, used, dt = oracle_rate(w, cpu_seconds, threads)
    # one host thread on the first 1e4 candidates (at most ~2 s of work)
    rate1, n1, _, dt1 = oracle_rate(w, 2.0, 1, max_n=10_000)
    out = {"workload": name, "candidates": n, "search": SEARCH_NAMES.get(search, search),
           "value": n / (ms / 1e3), "unit": UNIT, "ms_per_step": ms, "per_candidate_ns": 1e6 * ms / n,
           "step_ms": {"median": float(np.median(per)), "best": float(np.min(per)), "runs": len(per)},
           "single_batch_latency_ms": {"median": float(np.median(lat)), "best": float(np.min(lat)),
                                       "batch": batch},
           "l2": ("inputs %.1f MB; L2 flushed (256 MB write) before each timed step" % (in_bytes / 1e6)
                  if flush is not None else "inputs %.0f MB, larger than L2" % (in_bytes / 1e6)),
           "dominant_kernel": SEARCH_KERNELS.get(search, "search"),
           "roofline": {"bound": "alu", "achieved": tops, "peak": peak, "unit": "Tops/s",
                        "frac": tops / peak if tops else None,
                        "launch_us": 1e3 * s_ms / chunks, "launches_per_chunk": s_launches / chunks,
                        "phases_us_per_batch": {k: 1e3 * v[0] / chunks for k, v in ph.items()},
                        "ops_per_unit": OPS_PER_UNIT.get(search), "units_per_candidate": work["checks"] / n,
                        "searched_fraction": work["priced"] / n,
                        "upper_bound": search == 1},
           "device_errors": errors,
           "cpu_baseline": {"value": rate, "unit": UNIT, "cores": used, "kind": "oracle",
                            "sample": "first %d candidates (%.1f s, %d host threads)" % (ncpu, dt, used)},
           "cpu_single_thread": {"value": rate1, "unit": UNIT, "cores": 1, "kind": "oracle",
                                 "sample": "first %d candidates (%.2f s, one host thread)" % (n1, dt1)},
           "gpu_over_oracle": (n / (ms / 1e3)) / rate}
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--n", type=int, default=10_000_000)
    ap.add_argument("--batch", type=int, default=1_000_000)
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--mbs-levels", type=int, default=4, help="micro-batch sizes of the fill figure (0: skip)")
    ap.add_argument("--no-distribute", action="store_true", help="skip the paper's-split comparison figure")
    ap.add_argument("--plans", type=int, default=1_000_000, help="multi-template plans of the plan figure (0: skip)")
    ap.add_argument("--no-per-config", action="store_true", help="skip the per-workload measurements")
    ap.add_argument("--configs", default=",".join(PER_CONFIG),
                    help="comma-separated workloads of the per-workload measurements")
    ap.add_argument("--tiling", type=int, default=1_000_000,
                    help="moe48 candidates of the expert-tiling figure (0: skip)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))

    from paper_2609_34244_gb300 import workloads as W

    if args.impl == "reference":
        if rank != 0:
            return
        w = W.make_workload(WORKLOAD, seed=0, n=min(args.n, 400_000))
        print(json.dumps(run_reference(args, w)), flush=True)
        return

    import torch
    from paper_2609_34244_gb300 import _build
    _build.build()
    from paper_2609_34244_gb300 import heddle as h
    from paper_2609_34244_gb300 import shard

    torch.cuda.set_device(local)
    sms = torch.cuda.get_device_properties(local).multi_processor_count
    peaks, peak_kind = load_peaks()
    group = shard.init(world)
    n, batch = args.n, min(args.batch, args.n)
    # weak scaling: rank r prices its own n candidates (seed r), global indices r*n + c
    w = W.make_workload(WORKLOAD, seed=rank, n=n)
    base = rank * n
    ctx = h.heddle_create(local)
    h.heddle_load_cluster(ctx, w.cluster)
    h.heddle_load_model(ctx, w.model)
    h.heddle_set_chunk(ctx, batch)
    dc = h.cands_to_device(w.cands)
    res = h.alloc_results(n)
    state = h.alloc_topk_state()
    stream = torch.cuda.current_stream()
    cbatches = [(h.make_candidates(dc, lo, min(n, lo + batch), base_index=base),
                 h.make_results(res, lo, min(n, lo + batch))) for lo in range(0, n, batch)]
    n_batches = len(cbatches)
    call_all = h.make_candidates(dc, 0, n, base_index=base)
    res_all = h.make_results(res)

    def step():
        """One pass of the hot path: one heddle_price_topk call over all n
        candidates -- the library prices them in chunks of `batch` (screen,
        search) pipelined over four work streams and merges each chunk into
        the running top-16 in order."""
        h.heddle_topk_reset(ctx, state, 16, stream)
        h.heddle_price_topk(ctx, call_all, res_all, state, stream)

    search = h.heddle_get_search(ctx)

    def count_work():
        """Algorithmic work of one step (counting variant, untimed)."""
        for c, r in cbatches:
            h.heddle_count_next(ctx, True)
            h.heddle_price_candidates(ctx, c, r, stream)
        return h.heddle_work_counters(ctx)

    work = count_work()

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    shard.barrier(group)
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # per-kernel device time: the library records events around its screen,
    # search and top-k launches of every chunk while phase timing is on --
    # here on every PHASE_EVERY-th timed step (a sample: the events cost a
    # few per cent of the step), so `value` counts all steps at nearly full
    # speed while the kernels are still timed inside the timed region
    PHASE_EVERY = 8
    with ClockSampler(local) as clk:
        torch.cuda.synchronize()
        t_start.record(stream)
        step_ev = []
        sampled = 0
        for k in range(args.steps):
            timed = k % PHASE_EVERY == 0
            if timed:
                h.heddle_time_phases(ctx, True)
                sampled += 1
            step()
            if timed:
                h.heddle_time_phases(ctx, False)
            ev = torch.cuda.Event(enable_timing=True)
            ev.record(stream)
            step_ev.append(ev)
        t_end.record(stream)
        torch.cuda.synchronize()
    # per-step device times (consecutive events on the stream)
    step_ms = [t_start.elapsed_time(step_ev[0])] + [a.elapsed_time(b) for a, b in zip(step_ev, step_ev[1:])]
    shard.barrier(group)
    clocks = clk.summary()
    ms = t_start.elapsed_time(t_end)
    phases = h.heddle_phase_times(ctx)
    ms_all = shard.max_over_ranks(group, ms)
    errors = h.heddle_device_errors(ctx)
    local_topk = h.read_topk_state(state)
    merged = shard.merge_topk_across_ranks(group, local_topk, 16)

    # single-batch wall latency: one call on one batch of `batch` candidates,
    # host call to results ready (synchronised), after a warm call
    one_c, one_r = cbatches[0]
    h.heddle_topk_reset(ctx, state, 16, stream)
    h.heddle_price_topk(ctx, one_c, one_r, state, stream)
    torch.cuda.synchronize()
    lat = []
    for _ in range(20):
        t0 = time.perf_counter()
        h.heddle_topk_reset(ctx, state, 16, stream)
        h.heddle_price_topk(ctx, one_c, one_r, state, stream)
        torch.cuda.synchronize()
        lat.append((time.perf_counter() - t0) * 1e3)

    # the same kernels without overlap (one call per batch, so each chunk's
    # screen, search and top-k run alone): the search's isolated duration
    h.heddle_time_phases(ctx, True)
    for _ in range(3):
        h.heddle_topk_reset(ctx, state, 16, stream)
        for c, r in cbatches:
            h.heddle_price_topk(ctx, c, r, state, stream)
    torch.cuda.synchronize()
    h.heddle_time_phases(ctx, False)
    iso_phases = h.heddle_phase_times(ctx)

    # the paper's own layer split (§5.3) on the same candidates: its speed
    # and how much longer its iteration times are than the exact split's
    distribute = None
    if not args.no_distribute:
        res2 = h.alloc_results(n)
        res2_all = h.make_results(res2)
        h.heddle_set_search(ctx, h.SEARCH_DISTRIBUTE)
        dstate = h.alloc_topk_state()

        def dist_step():
            h.heddle_topk_reset(ctx, dstate, 16, stream)
            h.heddle_price_topk(ctx, call_all, res2_all, dstate, stream)

        dist_step()
        torch.cuda.synchronize()
        d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        d0.record(stream)
        for _ in range(2):
            dist_step()
        d1.record(stream)
        torch.cuda.synchronize()
        dms = d0.elapsed_time(d1) / 2
        ex_ok = res["status"] == 0
        di_ok = res2["status"] == 0
        both = ex_ok & di_ok
        gap = (res2["T"][both].double() - res["T"][both].double()) / res["T"][both].double()
        distribute = {"value": n / (dms / 1e3), "unit": UNIT, "ms_per_step": dms,
                      "exact_ok": int(ex_ok.sum()), "distribute_ok": int(di_ok.sum()),
                      "mean_T_gap_where_both_ok": float(gap.mean()) if both.any() else None,
                      "share_slower": float((gap > 0).double().mean()) if both.any() else None,
                      "share_faster": float((gap < 0).double().mean()) if both.any() else None,
                      "bottleneck_never_below_Bstar": bool((res2["bottleneck"][both] >= res["bottleneck"][both]).all())}
        h.heddle_set_search(ctx, h.SEARCH_AUTO)
        del res2

    # the general interval search on the same workload (secondary figure)
    general = None
    if search != h.SEARCH_GENERAL:
        h.heddle_set_search(ctx, h.SEARCH_GENERAL)
        gwork = count_work()
        for _ in range(2):
            step()
        torch.cuda.synchronize()
        g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        h.heddle_time_phases(ctx, True)
        g0.record(stream)
        for _ in range(2):
            step()
        g1.record(stream)
        torch.cuda.synchronize()
        h.heddle_time_phases(ctx, False)
        gms = g0.elapsed_time(g1) / 2
        gph = h.heddle_phase_times(ctx)
        gsearch_ms = gph["search"][0] / 2
        gtopk = h.read_topk_state(state)
        # the search kernels' own time: one call per batch, no overlap
        h.heddle_time_phases(ctx, True)
        h.heddle_topk_reset(ctx, state, 16, stream)
        for c, r in cbatches:
            h.heddle_price_topk(ctx, c, r, state, stream)
        torch.cuda.synchronize()
        h.heddle_time_phases(ctx, False)
        giso_ms = h.heddle_phase_times(ctx)["search"][0]
        general = {"value": n / (gms / 1e3), "ms_per_step": gms, "search_ms_per_step": gsearch_ms,
                   "search_us_per_batch_isolated": 1e3 * giso_ms / n_batches,
                   "checks_per_candidate": gwork["checks"] / n,
                   "probes_per_searched": gwork["probes"] / max(1, gwork["priced"]),
                   "alu_frac": gwork["checks"] * OPS_PER_UNIT[1] / (giso_ms / 1e3) / 1e12 /
                   (sms * LANES_PER_SM * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12),
                   "alu_frac_basis": "interval tests x 16 lane operations over the search kernels' "
                                     "isolated time (one call per batch)",
                   "same_topk": gtopk["idx"].tolist() == local_topk["idx"].tolist()}
        h.heddle_set_search(ctx, h.SEARCH_AUTO)

    # micro-batch-size fill (§5.3) on the same candidates: four sizes with
    # seeded per-size profiles, device-resident, timed like the main step
    mbs_fig = None
    if args.mbs_levels > 0:
        levels = args.mbs_levels
        h.heddle_load_mbs(ctx, levels, W.mbs_profiles(w, levels, seed=rank))
        mbs_out = torch.empty(n, dtype=torch.uint8, device="cuda")

        def mbs_step():
            for lo in range(0, n, batch):
                hi = min(n, lo + batch)
                h.heddle_price_mbs(ctx, h.make_candidates(dc, lo, hi, base_index=base),
                                   h.make_results(res, lo, hi), mbs_out[lo:hi], stream)

        for _ in range(2):
            mbs_step()
        torch.cuda.synchronize()
        m0, m1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        h.heddle_time_phases(ctx, True)
        m0.record(stream)
        for _ in range(3):
            mbs_step()
        m1.record(stream)
        torch.cuda.synchronize()
        h.heddle_time_phases(ctx, False)
        mph = h.heddle_phase_times(ctx)
        mms = m0.elapsed_time(m1) / 3
        ok = res["status"] == 0
        chosen = torch.bincount(mbs_out[ok].long(), minlength=levels).tolist()
        mbs_fig = {"value": n / (mms / 1e3), "unit": UNIT, "levels": levels, "ms_per_step": mms,
                   "phases_ms_per_step": {k: v[0] / 3 for k, v in mph.items()},
                   "ok_candidates_by_chosen_level": chosen,
                   "profiles": "seeded per-size profiles (workloads.mbs_profiles)"}
        h.heddle_load_mbs(ctx, 0)

    # multi-template plans (Algorithm 1): 1e6 plans of up to four templates
    # of the same workload, each template priced on the GPUs earlier ones left
    plans_fig = None
    if args.plans > 0:
        np_ = min(args.plans, 1 << 20)
        plans = W.make_plans(w, np_, 4, seed=rank)
        dp = h.plans_to_device(plans)
        pr = h.alloc_plan_results(np_, 4)
        h.heddle_price_plans(ctx, dp, pr, stream)
        torch.cuda.synchronize()
        p0, p1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        p0.record(stream)
        for _ in range(3):
            h.heddle_price_plans(ctx, dp, pr, stream)
        p1.record(stream)
        torch.cuda.synchronize()
        pms = p0.elapsed_time(p1) / 3
        plans_fig = {"value": np_ / (pms / 1e3), "unit": "plans/s", "plans_per_call": np_, "template_slots": 4,
                     "ms_per_call": pms,
                     "plans_by_templates_placed": torch.bincount(pr["placed"].long(), minlength=5).tolist(),
                     "best_plan_throughput": float(pr["thr"].max())}
        del dp, pr

    # expert tiling (§5.3) on the MoE workload: the same candidates priced
    # untiled and with every stage's EP x ETP x EDP choice, device-resident
    tiling_fig = None
    if args.tiling > 0:
        nt_ = args.tiling
        wt = W.make_workload("moe48", seed=rank, n=nt_)
        ctx2 = h.heddle_create(0)
        try:
            h.heddle_load_cluster(ctx2, wt.cluster)
            h.heddle_load_model(ctx2, wt.model)
            dct = h.cands_to_device(wt.cands)
            r_plain, r_tiled = h.alloc_results(nt_), h.alloc_results(nt_)
            til = torch.empty((32, nt_), dtype=torch.uint8, device="cuda")

            def timed(fn, reps=3):
                fn()
                torch.cuda.synchronize()
                e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                for _ in range(reps):
                    fn()
                e1.record(stream)
                torch.cuda.synchronize()
                return e0.elapsed_time(e1) / reps

            plain_ms = timed(lambda: h.heddle_price_candidates(ctx2, h.make_candidates(dct),
                                                               h.make_results(r_plain), stream))
            h.heddle_load_experts(ctx2, wt.model["expert_state_bytes"], wt.model["expert_param_bytes"])
            tiled_ms = timed(lambda: h.heddle_price_tiled(ctx2, h.make_candidates(dct), h.make_results(r_tiled),
                                                          til, stream))
            tiled_errors = h.heddle_device_errors(ctx2)
            pT, tT = r_plain["T"].cpu().numpy(), r_tiled["T"].cpu().numpy()
            pok, tok_ = r_plain["status"].cpu().numpy() == 0, r_tiled["status"].cpu().numpy() == 0
            both = pok & tok_
            codes = til.cpu().numpy()[:, tok_]
            Sk = wt.cands["S"][tok_]
            jk = (wt.cands["code"][:, tok_] >> 3) & 3
            layouts = {}
            for s_ in range(int(Sk.max()) if Sk.size else 0):
                live = Sk > s_
                le, lt = codes[s_, live] & 3, codes[s_, live] >> 2
                ld = jk[s_, live] - le - lt
                for a_, b_, c_ in zip(le, lt, ld):
                    key = "%dx%dx%d" % (1 << a_, 1 << b_, 1 << c_)
                    layouts[key] = layouts.get(key, 0) + 1
            ratio = tT[both].astype(np.float64) / pT[both].astype(np.float64)
            tiling_fig = {"value": nt_ / (tiled_ms / 1e3), "unit": UNIT, "workload": "moe48, %d candidates" % nt_,
                          "ms_per_call": tiled_ms, "untiled_ms_per_call": plain_ms,
                          "ok_untiled": int(pok.sum()), "ok_tiled": int(tok_.sum()),
                          "mean_T_ratio_tiled_over_untiled": float(ratio.mean()) if ratio.size else None,
                          "share_faster": float((ratio < 1).mean()) if ratio.size else None,
                          "share_slower": float((ratio > 1).mean()) if ratio.size else None,
                          "stage_layouts_EPxETPxEDP": dict(sorted(layouts.items(), key=lambda x: -x[1])),
                          "device_errors": int(tiled_errors)}
            del dct, r_plain, r_tiled, til
        finally:
            h.heddle_destroy(ctx2)

    # end to end through the public host-buffer call (pinned host memory,
    # placed on the GPU's own NUMA node: the process runs on the GPU's local
    # CPUs while the pages are pinned and first written)
    numa = gpu_numa(local)
    old_aff = os.sched_getaffinity(0) if hasattr(os, "sched_getaffinity") else None
    if numa.get("cpus") and old_aff is not None:
        try:
            os.sched_setaffinity(0, numa["cpus"])
        except OSError:
            pass
    pinned = {k: torch.empty(v.shape, dtype=torch.int16 if v.dtype == np.uint16 else torch.uint8, pin_memory=True)
              for k, v in w.cands.items()}
    for k, v in w.cands.items():
        pinned[k].numpy()[...] = v.view(np.int16) if v.dtype == np.uint16 else v
    copy_peak = h2d_copy_gbs(1 << 30)
    if old_aff is not None:
        try:
            os.sched_setaffinity(0, old_aff)
        except OSError:
            pass
    h2d = int(sum(v.numel() * v.element_size() for v in pinned.values()))
    st = h.new_topk_state(16)
    e2e_steps = max(1, args.e2e_steps)
    h.heddle_price_topk_host(ctx, pinned, None, st, batch, stream)  # warm (allocates staging)
    shard.barrier(group)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        st = h.new_topk_state(16)
        h.heddle_price_topk_host(ctx, pinned, None, st, batch, stream)
    e2e_s = (time.perf_counter() - t0) / e2e_steps
    e2e_s = shard.max_over_ranks(group, e2e_s)
    e2e_topk = h.topk_state_to_dict(st)
    h.heddle_destroy(ctx)

    if rank != 0:
        return
    per_config = None
    if not args.no_per_config:
        names = [x for x in args.configs.split(",") if x]
        unknown = sorted(set(names) - set(PER_CONFIG))
        if unknown:
            raise SystemExit("unknown workloads in --configs: %s" % ", ".join(unknown))
        per_config = [measure_config(h, name, peaks, sms) for name in names]
    value = n * world * args.steps / (ms_all / 1e3)
    ops_step = work["checks"] * OPS_PER_UNIT[search]
    peak_tops = sms * LANES_PER_SM * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    # the dominant kernel is the search: its average launch duration from
    # the events around it, its algorithmic ops per launch from the counters
    # per chunk: one screen launch per chunk (the equal-layer search is two
    # launches, its worklist pass and the pass over the entries it left open)
    search_ms, search_launches = phases["search"]
    chunks_timed = max(1, phases["screen"][1])
    search_us = 1e3 * search_ms / chunks_timed
    achieved_tops = ops_step * sampled / (search_ms / 1e3) / 1e12
    iso_ms, iso_launches = iso_phases["search"]
    iso_chunks = max(1, iso_phases["screen"][1])
    iso_tops = ops_step * 3 / (iso_ms / 1e3) / 1e12 if iso_ms > 0 else None
    total_phase_ms = sum(v[0] for v in phases.values())
    # the whole step against the same issue-slot peak: the screen's,
    # the search's and the top-k's algorithmic operations over the step time
    scr_ops = screen_ops(w.cands)
    tk_ops = TOPK_OPS_PER_SEARCHED * work["priced"]
    step_s = ms_all / args.steps / 1e3
    step_roofline = {"achieved": (scr_ops + ops_step + tk_ops) / step_s / 1e12, "peak": peak_tops,
                     "unit": "Tops/s", "frac": (scr_ops + ops_step + tk_ops) / step_s / 1e12 / peak_tops,
                     "ops_per_step": {"screen": scr_ops, "search": ops_step, "topk": tk_ops},
                     "screen_ops_basis": SCREEN_OPS, "topk_ops_per_searched": TOPK_OPS_PER_SEARCHED,
                     "how": "algorithmic lane operations of one step / the mean step time of the K timed steps"}
    cpu = None
    if not args.no_cpu_baseline:
        rate, ncpu, used, dt = oracle_rate(w, args.cpu_seconds, os.cpu_count() or 1)
        cpu = {"value": rate, "unit": UNIT, "cores": used, "kind": "oracle",
               "sample": "first %d candidates of %s seed 0 (%.1f s, %d host threads)" % (ncpu, WORKLOAD, dt, used)}
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_all / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": {"workload": WORKLOAD_DESC, "candidates_per_gpu": n, "batch": batch,
                   "parallelism": "candidate shards, dp%d" % world,
                   "l2": "inputs larger than L2 (%.0f MB of candidates per step per GPU)" % (h2d / 1e6),
                   "seed": "rank"},
        # per step the top-k reset kernel, plus the kernels the library
        # counted per step in the phase-timed steps (screen, search, top-k)
        "gpu_launches": (args.steps + args.steps * sum(v[1] for v in phases.values()) // max(1, sampled)) * world,
        "per_candidate_ns": 1e6 * ms_all / args.steps / n,
        "step_ms": {"median": float(np.median(step_ms)), "best": float(np.min(step_ms)),
                    "worst": float(np.max(step_ms)), "runs": len(step_ms)},
        "single_batch_latency_ms": {"median": float(np.median(lat)), "best": float(np.min(lat)),
                                    "batch": batch, "how": "wall time of one heddle_price_topk call on one batch, "
                                                           "synchronised, 20 runs after a warm call"},
        # the dominant kernel's own launch duration: one call per batch right
        # after the timed region, so no other chunk's kernel shares the GPU
        # with it; the overlapped launch time of the timed steps is under "live"
        "roofline": {"bound": "alu", "achieved": iso_tops, "peak": peak_tops, "unit": "Tops/s",
                     "frac": iso_tops / peak_tops if iso_tops else None,
                     "traffic": traffic_per_launch(search, batch),
                     "kernel": SEARCH_KERNELS[search], "search": SEARCH_NAMES[search],
                     "launch_us": 1e3 * iso_ms / iso_chunks, "chunks_timed": iso_chunks,
                     "launches_per_chunk": iso_launches / iso_chunks,
                     "duration_basis": "CUDA events around each chunk's search launches on their stream, one "
                                       "pricing call per batch (no overlap), 3 steps after the timed region",
                     "ops_per_unit": OPS_PER_UNIT[search],
                     "ops_per_launch": ops_step / n_batches,
                     "units_per_candidate": work["checks"] / n,
                     "probes_per_searched": work["probes"] / max(1, work["priced"]),
                     "searched_fraction": work["priced"] / n,
                     "phases_us_per_batch": {k: 1e3 * v[0] / iso_chunks for k, v in iso_phases.items()},
                     "live": {"launch_us": search_us, "chunks_timed": chunks_timed,
                              "achieved": achieved_tops, "frac": achieved_tops / peak_tops,
                              "phases_us_per_batch": {k: 1e3 * v[0] / chunks_timed for k, v in phases.items()},
                              "phase_share": {k: v[0] / total_phase_ms for k, v in phases.items()},
                              "how": "inside the timed steps (every 8th step): chunks pipelined over four work "
                                     "streams, so each launch shares the GPU with the neighbouring chunks' "
                                     "kernels"},
                     "step": step_roofline,
                     "peak_basis": "%s: %d SMs x %d lanes x %.0f MHz (%s sm_max)" % (
                         "issue slots", sms, LANES_PER_SM, float(peaks.get("sm_max_mhz", 2070.0)), peak_kind)},
        "clocks": clocks,
        "e2e": {"value": n * world / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d * world,
                "d2h_bytes_per_step": h.TOPK_STATE_BYTES * world,
                "d2h_contents": "the merged top-16 state (index, T and n*M of the 16 best plans); the per-candidate "
                                "T / n_dp / status planes stay on the device",
                "h2d_gbs_achieved": h2d / e2e_s / 1e9,
                "h2d_copy_peak_gbs": copy_peak,
                "copy_peak_how": "plain cudaMemcpyAsync of 1 GiB from pinned host memory, best of 5, CUDA events",
                "pinned_memory": {k: v for k, v in numa.items() if k != "cpus"}},
        "device_errors": errors,
        "general_search": general,
        "distribute_split": distribute,
        "mbs_fill": mbs_fig,
        "plans": plans_fig,
        "expert_tiling": tiling_fig,
        "per_config": per_config,
        "topk_head": merged["idx"][:4].tolist() if merged["count"] else [],
        "e2e_topk_matches": e2e_topk["idx"].tolist() == local_topk["idx"].tolist(),
    }
    if cpu:
        out["cpu_baseline"] = cpu
    print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
