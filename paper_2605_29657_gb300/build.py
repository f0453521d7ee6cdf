"""Builds liboccam.so (the C ABI of include/occam.h) for sm_103a with nvcc.

The translation units are compiled in parallel into ``_build/`` next to this
file and linked into ``liboccam.so`` in this package directory (both are
git-ignored build products). ``build(checked=True)`` makes the bounds-checked
variant instead (``-DOCCAM_CHECKED=1``: every computed gather, list and scan
index is tested in-kernel and a violation is recorded in the status word):
``liboccam_checked.so``, from ``_build_checked/``.
"""

from __future__ import annotations

import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
BUILD = os.path.join(HERE, "_build")
LIB = os.path.join(HERE, "liboccam.so")
LIB_CHECKED = os.path.join(HERE, "liboccam_checked.so")
SOURCES = ["stage1.cu", "stage1_tc.cu", "stage2.cu", "stage2_tc.cu", "stage2_scores_tc.cu", "compact.cu", "rules.cu", "selftest.cu", "api.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build liboccam.so")


def _flags():
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include")]


def build(verbose: bool = False, force: bool = False, checked: bool = False) -> str:
    """Builds liboccam.so (or, with checked, liboccam_checked.so) unless it
    is newer than every source. Concurrent callers (one per rank) serialise
    on a lock file."""
    import fcntl

    bdir = BUILD + ("_checked" if checked else "")
    os.makedirs(bdir, exist_ok=True)
    with open(os.path.join(bdir, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        try:
            return _build(verbose, force, checked)
        finally:
            fcntl.flock(lk, fcntl.LOCK_UN)


def _build(verbose: bool, force: bool, checked: bool = False) -> str:
    BUILD_DIR = BUILD + ("_checked" if checked else "")
    LIB_OUT = LIB_CHECKED if checked else LIB
    extra = ["-DOCCAM_CHECKED=1"] if checked else []
    nv = nvcc()
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(ROOT, "include", "occam.h")]
    newest = max(os.path.getmtime(d) for d in deps)
    if not force and os.path.exists(LIB_OUT) and os.path.getmtime(LIB_OUT) >= newest and os.path.getmtime(LIB_OUT) >= os.path.getmtime(__file__):
        return LIB_OUT
    procs = []
    objs = []
    for src in SOURCES:
        obj = os.path.join(BUILD_DIR, src.replace(".cu", ".o"))
        objs.append(obj)
        cmd = [nv] + _flags() + extra + ["-Xptxas", "-v", "-c", os.path.join(CSRC, src), "-o", obj]
        log = open(os.path.join(BUILD_DIR, src.replace(".cu", ".log")), "w")
        procs.append((src, subprocess.Popen(cmd, stdout=log, stderr=subprocess.STDOUT), log))
    failed = []
    for src, p, log in procs:
        rc = p.wait()
        log.close()
        if rc != 0:
            failed.append(src)
    if failed:
        msgs = "".join(open(os.path.join(BUILD_DIR, s.replace(".cu", ".log"))).read()[-3000:] for s in failed)
        raise RuntimeError(f"nvcc failed for {failed}:\n{msgs}")
    tmp = LIB_OUT + ".tmp"
    cmd = [nv] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + objs + ["-ldl"]
    subprocess.run(cmd, check=True, capture_output=not verbose)
    os.replace(tmp, LIB_OUT)
    if verbose:
        print("built", LIB_OUT, file=sys.stderr)
    return LIB_OUT


if __name__ == "__main__":
    build(verbose=True, force="--force" in sys.argv, checked="--checked" in sys.argv)
