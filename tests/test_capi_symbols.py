"""The C-ABI library builds, loads without a GPU and exports every function
include/heddle.h declares; the ctypes structs match the C layouts."""

import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "heddle.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(heddle_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for n in ("heddle_load_cluster", "heddle_load_model", "heddle_price_candidates", "heddle_topk"):
        assert n in names


def test_library_exports_every_declared_symbol(heddle_lib):
    L = heddle_lib.load_library()
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing
    assert sorted(heddle_lib.EXPORTS) == declared_functions()
    out = subprocess.run(["nm", "-D", "--defined-only", heddle_lib.LIB_PATH], capture_output=True,
                         text=True).stdout
    for n in declared_functions():
        assert re.search(r"\bT %s$" % n, out, re.M), n


def test_struct_layouts_match_header(heddle_lib, tmp_path):
    import ctypes as C
    src = tmp_path / "sz.c"
    src.write_text(r'''
#include <stdio.h>
#include <stddef.h>
#include "heddle.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu\n", sizeof(heddle_gpu_type), sizeof(heddle_node), sizeof(heddle_layer),
         sizeof(heddle_candidates), sizeof(heddle_results), sizeof(heddle_topk_state));
  printf("%zu %zu %zu %zu\n", offsetof(heddle_candidates, base_index), offsetof(heddle_topk_state, idx),
         offsetof(heddle_topk_state, T), offsetof(heddle_topk_state, nM));
  return 0;
}''')
    exe = tmp_path / "sz"
    subprocess.check_call(["gcc", "-std=c11", "-I", os.path.join(ROOT, "include"), str(src), "-o", str(exe)])
    lines = subprocess.check_output([str(exe)], text=True).split("\n")
    h = heddle_lib
    sizes = [C.sizeof(t) for t in (h.heddle_gpu_type, h.heddle_node, h.heddle_layer, h.heddle_candidates,
                                   h.heddle_results, h.heddle_topk_state)]
    assert [int(v) for v in lines[0].split()] == sizes
    offs = [h.heddle_candidates.base_index.offset, h.heddle_topk_state.idx.offset,
            h.heddle_topk_state.T.offset, h.heddle_topk_state.nM.offset]
    assert [int(v) for v in lines[1].split()] == offs


def test_create_without_gpu_fails_loudly(heddle_lib):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(heddle_lib.HeddleError):
        heddle_lib.heddle_create(0)


def test_missing_library_fails_loudly(tmp_path):
    # the binding has no fallback: without the built library every entry
    # point raises instead of computing anything
    import sys
    code = ("from paper_2609_34244_gb300 import heddle as h\n"
            "try:\n"
            "    h.heddle_create(0)\n"
            "except RuntimeError as e:\n"
            "    print('raised:', e)\n")
    env = dict(os.environ, HEDDLE_LIB=str(tmp_path / "libheddle.so"))
    p = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=300)
    assert p.returncode == 0, p.stderr[-2000:]
    assert "raised:" in p.stdout and "not built" in p.stdout
