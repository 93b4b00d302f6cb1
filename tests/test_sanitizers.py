"""The oracle and the C ABI's host code under AddressSanitizer and
UndefinedBehaviorSanitizer (CPU, no GPU).

The oracle is rebuilt with -fsanitize=address,undefined and every one of its
entry points runs on small seeded workloads in a child process (the ASan
runtime preloaded); any report fails the child, and its results must equal
the plain build's.  The CUDA library is rebuilt with its host code
instrumented the same way; the host-side checks that run without a device
(missing context, argument and limit checks of the allocation-free top-k,
context creation on a machine without a GPU) run in a child under the
sanitizers.  The host paths that need a device are covered by the GPU tests,
not here."""

import os
import subprocess
import sys

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
SAN = ["-fsanitize=address,undefined", "-fno-sanitize-recover=all", "-fno-omit-frame-pointer"]


def _runtime():
    p = subprocess.run(["gcc", "-print-file-name=libasan.so"], capture_output=True, text=True)
    path = p.stdout.strip()
    if p.returncode != 0 or not os.path.isabs(path) or not os.path.exists(path):
        pytest.skip("no AddressSanitizer runtime for gcc here")
    return path


def _env(extra):
    env = dict(os.environ)
    env.update(extra)
    env["LD_PRELOAD"] = _runtime()
    env["ASAN_OPTIONS"] = "detect_leaks=0:halt_on_error=1:abort_on_error=0"
    env["UBSAN_OPTIONS"] = "halt_on_error=1:print_stacktrace=1"
    return env


def test_oracle_under_asan_ubsan(tmp_path):
    lib = str(tmp_path / "liboracle_san.so")
    src = os.path.join(ROOT, "oracle", "heddle_oracle.c")
    subprocess.check_call(["gcc", "-std=c11", "-O1", "-g", "-ffp-contract=off", "-fPIC", "-shared", *SAN,
                           "-o", lib, src, "-lpthread", "-lm"])
    out_san = str(tmp_path / "san.npz")
    p = subprocess.run([sys.executable, os.path.join(HERE, "sanitize_child.py"), "oracle", out_san],
                       env=_env({"HEDDLE_ORACLE_LIB": lib}), capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stdout[-2000:] + p.stderr[-4000:]
    assert "ERROR: AddressSanitizer" not in p.stderr and "runtime error" not in p.stderr, p.stderr[-4000:]
    out_plain = str(tmp_path / "plain.npz")
    env = dict(os.environ)
    env.pop("HEDDLE_ORACLE_LIB", None)
    subprocess.check_call([sys.executable, os.path.join(HERE, "sanitize_child.py"), "oracle", out_plain], env=env,
                          timeout=600)
    a, b = np.load(out_san), np.load(out_plain)
    assert sorted(a.files) == sorted(b.files)
    for k in a.files:
        assert np.array_equal(a[k], b[k]), k


def test_capi_host_code_under_asan_ubsan():
    from paper_2609_34244_gb300 import _build
    lib = _build.build(variant="asan")
    p = subprocess.run([sys.executable, os.path.join(HERE, "sanitize_child.py"), "capi"],
                       env=_env({"HEDDLE_LIB": lib}), capture_output=True, text=True, timeout=600)
    if p.returncode != 0 and "CUDA driver" in p.stderr and "capi ok" not in p.stdout:
        pytest.fail(p.stderr[-3000:])
    assert p.returncode == 0 and "capi ok" in p.stdout, p.stdout[-2000:] + p.stderr[-4000:]
    assert "ERROR: AddressSanitizer" not in p.stderr and "runtime error" not in p.stderr, p.stderr[-4000:]


def test_harness_reports_a_planted_overflow(tmp_path):
    """The same flags and environment catch a heap overflow planted in a
    small host library, so a clean run above means something."""
    src = tmp_path / "planted.c"
    src.write_text("#include <stdlib.h>\nint planted(int i) { int* p = malloc(4 * sizeof(int)); int v = p[i]; "
                   "free(p); return v; }\n")
    lib = str(tmp_path / "libplanted.so")
    subprocess.check_call(["gcc", "-O1", "-g", "-fPIC", "-shared", *SAN, "-o", lib, str(src)])
    code = "import ctypes, sys; ctypes.CDLL(sys.argv[1]).planted(4)"
    p = subprocess.run([sys.executable, "-c", code, lib], env=_env({}), capture_output=True, text=True, timeout=120)
    assert p.returncode != 0, p.stderr[-2000:]
    assert "heap-buffer-overflow" in p.stderr or "runtime error" in p.stderr, p.stderr[-2000:]
