"""Builds liboccam.so (the C ABI of include/occam.h) for sm_103a with nvcc.

The translation units are compiled in parallel into ``_build/`` next to this
file and linked into ``liboccam.so`` in this package directory (both are
git-ignored build products).
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
SOURCES = ["stage1.cu", "stage1_tc.cu", "stage2.cu", "stage2_tc.cu", "stage2_scores_tc.cu", "compact.cu", "rules.cu", "selftest.cu", "api.cu"]
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    for cand in (os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"):
        if cand and os.path.exists(cand):
            return cand
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build liboccam.so")


def _flags():
    return ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC", "-I", os.path.join(ROOT, "include")]


def build(verbose: bool = False, force: bool = False) -> str:
    """Builds liboccam.so unless it is newer than every source. Concurrent
    callers (one per rank) serialise on a lock file."""
    import fcntl

    os.makedirs(BUILD, exist_ok=True)
    with open(os.path.join(BUILD, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        try:
            return _build(verbose, force)
        finally:
            fcntl.flock(lk, fcntl.LOCK_UN)


def _build(verbose: bool, force: bool) -> str:
    nv = nvcc()
    deps = [os.path.join(CSRC, f) for f in os.listdir(CSRC)] + [os.path.join(ROOT, "include", "occam.h")]
    newest = max(os.path.getmtime(d) for d in deps)
    if not force and os.path.exists(LIB) and os.path.getmtime(LIB) >= newest and os.path.getmtime(LIB) >= os.path.getmtime(__file__):
        return LIB
    procs = []
    objs = []
    for src in SOURCES:
        obj = os.path.join(BUILD, src.replace(".cu", ".o"))
        objs.append(obj)
        cmd = [nv] + _flags() + ["-Xptxas", "-v", "-c", os.path.join(CSRC, src), "-o", obj]
        log = open(os.path.join(BUILD, src.replace(".cu", ".log")), "w")
        procs.append((src, subprocess.Popen(cmd, stdout=log, stderr=subprocess.STDOUT), log))
    failed = []
    for src, p, log in procs:
        rc = p.wait()
        log.close()
        if rc != 0:
            failed.append(src)
    if failed:
        msgs = "".join(open(os.path.join(BUILD, s.replace(".cu", ".log"))).read()[-3000:] for s in failed)
        raise RuntimeError(f"nvcc failed for {failed}:\n{msgs}")
    tmp = LIB + ".tmp"
    cmd = [nv] + ARCH + ["-shared", "-cudart", "shared", "-o", tmp] + objs
    subprocess.run(cmd, check=True, capture_output=not verbose)
    os.replace(tmp, LIB)
    if verbose:
        print("built", LIB, file=sys.stderr)
    return LIB


if __name__ == "__main__":
    build(verbose=True, force="--force" in sys.argv)
