"""bench.py's host side, run here without a GPU: the reference arm (the CPU
oracle on a bounded sample per step) prints one JSON line carrying the
benchmark contract's keys and an e2e object with no copied bytes, and
nothing on a rank other than 0; the screen's algorithmic operation count
and the clock record's parsing (median, maximum, active throttle reasons)
are recomputed by hand."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(args, env_extra=None):
    env = dict(os.environ)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, env=env,
                          capture_output=True, text=True, timeout=900)


def test_reference_arm_prints_one_contract_line(oracle_mod):
    p = _run(["--impl", "reference", "--steps", "1", "--warmup", "3"])
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [line for line in p.stdout.splitlines() if line.startswith("{")]
    assert len(lines) == 1, p.stdout[-2000:]
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference"
    assert (d["n_gpus"], d["steps"], d["warmup"]) == (1, 1, 3)
    assert d["unit"] == "candidates/s" and d["higher_is_better"] is True and d["value"] > 0
    assert d["ms_per_step"] > 0 and d["vs_baseline"] is None
    assert d["config"]["candidates_per_step"] > 0 and "workload" in d["config"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_arm_other_ranks_print_nothing():
    p = _run(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"],
             {"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"})
    assert p.returncode == 0, p.stderr[-2000:]
    assert not p.stdout.strip()


def _bench_module():
    import importlib.util
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_screen_ops_counts_per_candidate_stage_type_and_pair():
    # the screen's algorithmic count, recounted candidate by candidate
    from paper_2609_34244_gb300 import workloads as W
    b = _bench_module()
    cands = W.make_workload("dense80", seed=3, n=500).cands
    exp = 0
    for c in range(cands["S"].shape[0]):
        S = int(cands["S"][c])
        codes = [int(cands["code"][s, c]) for s in range(S)]
        exp += (b.SCREEN_OPS["candidate"] + b.SCREEN_OPS["stage"] * S
                + b.SCREEN_OPS["type"] * len({x & 7 for x in codes})
                + b.SCREEN_OPS["pair"] * len({x & 31 for x in codes}))
    assert b.screen_ops(cands) == exp


def test_clock_summary_reads_median_max_and_active_reasons(tmp_path):
    b = _bench_module()
    csv = tmp_path / "clocks.csv"
    csv.write_text("0, 2070, 2070, 900.1, 0x4, Not Active, Not Active, Not Active, Active\n"
                   "0, 1980, 2070, 950.3, 0x4, Not Active, Not Active, Not Active, Active\n"
                   "0, 2055, 2070, 910.0, 0x0, Not Active, Active, Not Active, Not Active\n"
                   "garbled line\n")
    s = b.ClockSampler(0)
    s.path = str(csv)
    out = s.summary()
    assert out == {"sm_mhz": 2055.0, "sm_max_mhz": 2070.0,
                   "reasons": ["hw_thermal_slowdown", "sw_power_cap"], "samples": 3}
    empty = b.ClockSampler(0)
    assert empty.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
