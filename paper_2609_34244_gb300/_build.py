"""Build ``libheddle.so`` in-tree with nvcc for sm_103a (GB300).

Each ``csrc/*.cu`` translation unit compiles in parallel to an object file
under ``_build/``; the objects link into ``paper_2609_34244_gb300/libheddle.so``
(CUDA runtime linked statically).  Rebuilds only when a source or header is
newer than the library.  Works without a GPU (cross-compilation).
"""

from __future__ import annotations

import concurrent.futures as cf
import glob
import os
import shutil
import subprocess

PKG = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(PKG)
CSRC = os.path.join(PKG, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(ROOT, "_build")
LIB = os.path.join(PKG, "libheddle.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
NVCC_FLAGS = ["-O3", "-std=c++17", "-lineinfo", "-Xcompiler", "-fPIC", "-Xcompiler", "-O2",
              "-I", INCLUDE, "-I", CSRC]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libheddle.so")


def _sources():
    return sorted(glob.glob(os.path.join(CSRC, "*.cu")))


def _deps():
    return _sources() + glob.glob(os.path.join(CSRC, "*.cuh")) + glob.glob(os.path.join(INCLUDE, "*.h")) \
        + [os.path.abspath(__file__)]


# Variants of the library beside the product build, for the tests:
# "checked" adds device-side bounds checks that raise an error flag instead of
# reading or writing out of range, and shrinks the equal-layer search's queue
# of open searches so its fallback path runs often; "asan" instruments the
# host code with AddressSanitizer and UndefinedBehaviorSanitizer.
VARIANTS = {
    "checked": ["-DHEDDLE_CHECKED=1"],
    "asan": ["-Xcompiler", "-fsanitize=address", "-Xcompiler", "-fsanitize=undefined", "-Xcompiler",
             "-fno-omit-frame-pointer", "-Xcompiler", "-fno-sanitize-recover=all"],
}

VARIANT_LINK = {"asan": ["-Xcompiler", "-fsanitize=address", "-Xcompiler", "-fsanitize=undefined"]}


def lib_path(variant: str | None = None) -> str:
    return LIB if not variant else os.path.join(PKG, "libheddle_%s.so" % variant)


def stale(variant: str | None = None) -> bool:
    path = lib_path(variant)
    if not os.path.exists(path):
        return True
    t = os.path.getmtime(path)
    return any(os.path.getmtime(p) > t for p in _deps())


def build(force: bool = False, verbose: bool = False, extra: list | None = None, variant: str | None = None) -> str:
    """Compile and link; returns the library path (``variant``: one of
    VARIANTS, built beside the product library)."""
    target = lib_path(variant)
    if not force and not stale(variant):
        return target
    objdir = BUILD if not variant else os.path.join(BUILD, variant)
    os.makedirs(objdir, exist_ok=True)
    cc = nvcc()
    extra = list(extra or []) + (VARIANTS[variant] if variant else [])

    def compile_one(src):
        obj = os.path.join(objdir, os.path.basename(src) + ".o")
        cmd = [cc, *ARCH, *NVCC_FLAGS, *extra, "-c", src, "-o", obj]
        p = subprocess.run(cmd, capture_output=True, text=True)
        if p.returncode != 0:
            raise RuntimeError("nvcc failed for %s:\n%s\n%s" % (src, " ".join(cmd), p.stderr))
        return obj, p.stderr

    with cf.ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        results = list(ex.map(compile_one, _sources()))
    if verbose:
        for obj, err in results:
            if err.strip():
                print(err)
    tmp = target + ".tmp%d" % os.getpid()
    link_extra = VARIANT_LINK.get(variant, [])
    cmd = [cc, *ARCH, "-shared", "-o", tmp, *[o for o, _ in results], "-cudart", "static", *link_extra]
    p = subprocess.run(cmd, capture_output=True, text=True)
    if p.returncode != 0:
        raise RuntimeError("link failed:\n%s\n%s" % (" ".join(cmd), p.stderr))
    os.replace(tmp, target)
    return target


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose=True,
                extra=["-Xptxas", "-v"] if "--ptxas" in sys.argv else None))
