"""The pins must catch plausible mistakes in the oracle.

Each mutant is a temporary copy of ``oracle/heddle_oracle.c`` with one
planted mistake (a dropped term, a wrong comparison, index or operand); it is
compiled on the CPU into a temporary directory and the full pin suite of
``pin_checks.py`` runs against it in a child process.  Every mutant must fail
at least one pin.  The committed oracle is never modified.
"""

import json
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "heddle_oracle.c")

MUTANTS = [
    ("drop_p2p_in_dp", "int64_t t = P[s][j] - P[s][i] + c[s];", "int64_t t = P[s][j] - P[s][i];"),
    ("memory_strict", "if (W[s][j] - W[s][i] > cap[s]) continue;\n                int64_t t",
     "if (W[s][j] - W[s][i] >= cap[s]) continue;\n                int64_t t"),
    ("iteration_M_not_M_minus_1", "return (int64_t)(M - 1) * tmax", "return (int64_t)M * tmax"),
    ("drop_grad_sync", "+ tsum + gmax;", "+ tsum;"),
    ("drop_sum_term", "return (int64_t)(M - 1) * tmax + tsum + gmax;",
     "return (int64_t)(M - 1) * tmax + tmax + gmax;"),
    ("inflight_reversed", "int64_t inflight = (S - s) < M ? (S - s) : M;",
     "int64_t inflight = (s + 1) < M ? (s + 1) : M;"),
    ("inflight_ignores_M", "int64_t inflight = (S - s) < M ? (S - s) : M;",
     "int64_t inflight = (S - s);"),
    ("tp_ring_factor", "double ring = (2.0 * (k - 1.0)) / k;", "double ring = (k - 1.0) / k;"),
    ("ep_factor", "t = 4.0 * part;", "t = 2.0 * part;"),
    ("collective_bw_rule", "(1 << j) <= x->maxnode[g] ? (double)x->intra_bw[g]",
     "(1 << j) < x->maxnode[g] ? (double)x->intra_bw[g]"),
    ("p2p_same_node_rule", "(1 << j[s]) + (1 << j[s + 1]) <= x->maxnode[g[s]]",
     "(1 << j[s]) + (1 << j[s + 1]) < x->maxnode[g[s]]"),
    ("p2p_direction", "c[s] = x->p2p[g[s]][g[s + 1]][same];", "c[s] = x->p2p[g[s]][g[s]][same];"),
    ("dp_ring_factor", "u128 num = (u128)2 * (u128)(n - 1)", "u128 num = (u128)(n - 1)"),
    ("dp_shard_not_divided", "u128 den = (u128)n * (u128)(1 << j[s]) *", "u128 den = (u128)n *"),
    ("walk_ignores_remainder", "if (F(s + 1, j) > B) continue;", ""),
    ("round_truncates", "return (int64_t)llround(seconds * 1e9);", "return (int64_t)(seconds * 1e9);"),
    ("ffd_increasing", "for (int e = 3; e >= 0 && ok; --e)", "for (int e = 0; e <= 3 && ok; ++e)"),
    ("topk_tie_larger_index", "return a->idx < b->idx ? -1 : (a->idx > b->idx ? 1 : 0);",
     "return a->idx > b->idx ? -1 : (a->idx < b->idx ? 1 : 0);"),
    ("rank_operand_transposed", "u128 lhs = (u128)a->nM * (u128)b->T;", "u128 lhs = (u128)a->nM * (u128)a->T;"),
    ("mem_cap_not_times_k", "cap[s] = x->mem[g[s]] * (int64_t)(1 << j[s]);", "cap[s] = x->mem[g[s]];"),
    ("nic_max_not_min", "if (node_nic[b] < x->inter_bw[g]) x->inter_bw[g] = node_nic[b];",
     "if (x->inter_bw[g] == INT64_MAX || node_nic[b] > x->inter_bw[g]) x->inter_bw[g] = node_nic[b];"),
    ("ceil_is_floor", "return (int64_t)((a + b - 1) / b);", "return (int64_t)(a / b);"),
    ("tp_mask_off_by_one", "(!x->moe && (1 << j[s]) > x->maxnode[g[s]])",
     "(!x->moe && (1 << j[s]) >= x->maxnode[g[s]])"),
    ("empty_stage_allowed", "for (int j = i + 1; j <= L; ++j) {\n                if (F(s + 1, j) == INF) continue;",
     "for (int j = i; j <= L; ++j) {\n                if (F(s + 1, j) == INF) continue;"),
    ("max_not_min_in_dp", "if (v < best) best = v;", "if (best == INF || v > best) best = v;"),
    ("ep_group_not_split", "while ((1 << e) > x->maxnode[t]) --e;", ""),
    ("ep_blocks_of_one", "while ((1 << e) > x->maxnode[t]) --e;", "if ((1 << e) > x->maxnode[t]) e = 0;"),
    ("compute_ignores_degree", "double s = flops / (k * tflops * 1e12);", "double s = flops / (tflops * 1e12);"),
    ("distribute_tie_to_later", "if (!given[s] && (best < 0 || rem[s] > rem[best])) best = s;",
     "if (!given[s] && (best < 0 || rem[s] >= rem[best])) best = s;"),
    ("distribute_no_one_layer_minimum", "if (cnt[s] < 1) cnt[s] = 1;", "if (cnt[s] < 0) cnt[s] = 0;"),
    ("distribute_time_not_speed", "w[0][s] = all > 0 ? ((int64_t)1 << 40) / all : ((int64_t)1 << 40);",
     "w[0][s] = all;"),
    ("distribute_memory_ignored", "if (W[s][b[s + 1]] - W[s][b[s]] > cap[s]) fits = 0;", "(void)cap;"),
    ("plans_first_fit_not_exact_size", "if (x->node_type[d] == g[s] && node_free[d] == w) {",
     "if (x->node_type[d] == g[s] && node_free[d] >= w) {"),
    ("plans_continue_after_failure", "                ended = 1;\n                continue;",
     "                continue;"),
    ("plans_degree_from_whole_cluster", "price_one(x, St, M[o], codes, f, Wbuf, &r, node_free);",
     "price_one(x, St, M[o], codes, f, Wbuf, &r, NULL);"),
    ("plans_throughput_per_ns", "sum = sum + ((double)(r.n * (int64_t)M[o]) * 1e9) / (double)r.T;",
     "sum = sum + ((double)(r.n * (int64_t)M[o])) / (double)r.T;"),
    ("distribute_choice_sees_gradient", "int64_t pipe = (int64_t)(M - 1) * tmax + tsum;",
     "int64_t tm2, pipe = evaluate(x, S, M, n, P, c, j, g, b, &tm2);"),
    ("tiling_etp_leaves_node", "x->tvalid[g][slot] = x->gpus[g] > 0 && (1 << lt) <= x->maxnode[g];",
     "x->tvalid[g][slot] = x->gpus[g] > 0;"),
    ("tiling_ep_group_without_etp", "double bw = (1 << (le + lt)) <= x->maxnode[g] ? near : far;",
     "double bw = (1 << le) <= x->maxnode[g] ? near : far;"),
    ("tiling_etp_ring_factor", "sec = sec + ((4.0 * ((2.0 * (t - 1.0)) / t)) * (double)x->a2a[l]) / near;",
     "sec = sec + ((4.0 * ((t - 1.0) / t)) * (double)x->a2a[l]) / near;"),
    ("tiling_split_ignores_edp_memory", "int64_t mem = (x->state[j] - x->state[i]) + tl->d1[o] * (x->estate[j] - x->estate[i]) +",
     "int64_t mem = (x->state[j] - x->state[i]) + 0 * (x->estate[j] - x->estate[i]) +"),
    ("tiling_choice_ignores_memory", "fits[s][o] = mem <= cap[s];", "fits[s][o] = 1;"),
    ("tiling_sync_ignores_edp", "(u128)(n * d - 1) * (u128)Ge", "(u128)(n - 1) * (u128)Ge"),
    ("tiling_sync_always_nic", "int64_t bw = (n == 1 && (1 << j) <= x->maxnode[g]) ? x->intra_bw[g] : x->inter_bw[g];",
     "int64_t bw = x->inter_bw[g];"),
    ("tiling_no_reselection", "if (fits[s][o] && og[s][o] <= Y && (pick[s] < 0", "if (fits[s][o] && (pick[s] < 0"),
    ("tiling_tie_to_later_slot", "(pick[s] < 0 || ot[s][o] < ot[s][pick[s]])", "(pick[s] < 0 || ot[s][o] <= ot[s][pick[s]])"),
    ("tiling_edp_order_reversed", "    for (int d = 0; d <= j; ++d)\n        for (int t = 0; t + d <= j; ++t) {",
     "    for (int d = j; d >= 0; --d)\n        for (int t = 0; t + d <= j; ++t) {"),
]

# planted mistakes in the Python part of the oracle (the micro-batch fill)
PY_SRC = os.path.join(ROOT, "oracle", "oracle.py")
PY_MUTANTS = [
    ("mbs_flops_not_scaled", 'out["flops"] = np.asarray(model["flops"], np.float64) * float(f)',
     'out["flops"] = np.asarray(model["flops"], np.float64)'),
    ("mbs_act_not_scaled", 'for k in ("act_bytes", "ar_bytes", "a2a_bytes"):', 'for k in ("ar_bytes", "a2a_bytes"):'),
    ("mbs_boundary_not_scaled", 'out["boundary_bytes"] = int(model["boundary_bytes"]) * f',
     'out["boundary_bytes"] = int(model["boundary_bytes"])'),
    ("mbs_tie_to_larger", '(r["T"] < best["T"])', '(r["T"] <= best["T"])'),
    ("mbs_no_divisibility", 'ci["M"] = np.where(div, M >> i, 0).astype(np.uint16)',
     'ci["M"] = np.maximum(M >> i, 1).astype(np.uint16)'),
    ("mbs_M_not_divided", "np.where(div, M >> i, 0)", "np.where(div, M, 0)"),
]

CHILD = r"""
import json, sys, traceback, types
sys.path[:0] = [sys.argv[1], sys.argv[1] + "/tests"]
from oracle import oracle as O
if len(sys.argv) > 3:
    # a planted mistake in oracle.py: run the mutated source as the module
    M = types.ModuleType("oracle_mutant")
    M.__dict__["__file__"] = O.__file__
    exec(compile(open(sys.argv[3]).read(), O.__file__, "exec"), M.__dict__)
    O = M
O.LIB = sys.argv[2]
O.build = lambda force=False: O.LIB
import pin_checks as P
failed = []
for chk in P.ALL_CHECKS:
    try:
        chk(O)
    except Exception as e:
        failed.append(chk.__name__)
print("FAILED=" + json.dumps(failed))
"""


def _compile(dirpath, text):
    src = os.path.join(dirpath, "heddle_oracle.c")
    with open(src, "w") as f:
        f.write(text)
    shutil.copy(os.path.join(ROOT, "oracle", "heddle_oracle.h"), dirpath)
    lib = os.path.join(dirpath, "libmutant.so")
    subprocess.check_call(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared",
                           "-o", lib, src, "-lpthread", "-lm"])
    return lib


def _run_pins(lib, py_src=None):
    try:
        p = subprocess.run([sys.executable, "-c", CHILD, ROOT, lib] + ([py_src] if py_src else []),
                           capture_output=True, text=True, timeout=300)
    except subprocess.TimeoutExpired:
        return ["<timeout>"]
    for line in p.stdout.splitlines():
        if line.startswith("FAILED="):
            return json.loads(line[len("FAILED="):])
    return ["<crash rc=%d>" % p.returncode]


def test_unmutated_copy_passes(tmp_path):
    with open(SRC) as f:
        text = f.read()
    assert _run_pins(_compile(str(tmp_path), text)) == []


@pytest.mark.parametrize("name,old,new", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_mutant_is_caught(tmp_path, name, old, new):
    with open(SRC) as f:
        text = f.read()
    assert text.count(old) == 1, "mutation site not unique: " + name
    failed = _run_pins(_compile(str(tmp_path), text.replace(old, new)))
    assert failed, "no pin catches mutant " + name


@pytest.mark.parametrize("name,old,new", PY_MUTANTS, ids=[m[0] for m in PY_MUTANTS])
def test_python_mutant_is_caught(tmp_path, name, old, new):
    with open(SRC) as f:
        lib = _compile(str(tmp_path), f.read())
    with open(PY_SRC) as f:
        text = f.read()
    assert text.count(old) == 1, "mutation site not unique: " + name
    py = os.path.join(str(tmp_path), "oracle_mutant.py")
    with open(py, "w") as f:
        f.write(text.replace(old, new))
    failed = _run_pins(lib, py)
    assert failed, "no pin catches mutant " + name
