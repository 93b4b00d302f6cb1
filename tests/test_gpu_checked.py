"""The bounds-checked build (HEDDLE_CHECKED): every data-dependent index the
kernels use -- worklist entries, candidate indices, table rows -- is tested
before use, and a failed test raises a device flag and skips the access
instead of trapping.  Seeded workloads in every search mode, through it,
must match the oracle with no flag raised.  Runs in a child process, which
loads the checked library in place of the product one."""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


def test_checked_build_matches_oracle_without_flags(oracle_mod):
    from paper_2609_34244_gb300 import _build
    lib = _build.build(variant="checked")
    env = dict(os.environ)
    env["HEDDLE_LIB"] = lib
    p = subprocess.run([sys.executable, os.path.join(HERE, "checked_child.py")], env=env, capture_output=True,
                       text=True, timeout=1200)
    assert p.returncode == 0 and "checked ok" in p.stdout, p.stdout[-3000:] + p.stderr[-3000:]
