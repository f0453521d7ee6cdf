"""The bounds-checked build (OCCAM_CHECKED=1) on a representative set of the
parity cases: fused Stage II with 4-, 8- and 16-CTA clusters, the two-pass
kernels, mutual Stage I, compaction and the no-allocation entry point. Every
computed gather, list and scan index is tested in-kernel; the cases must end
with device status 0 and still match the oracle. The checked library is
built on demand and loaded in a process of its own."""

from __future__ import annotations

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_checked_build_parity():
    from paper_2605_29657_gb300 import build as pb

    pb.build(checked=True)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "tests", "_checked_cases.py")], cwd=ROOT,
                       capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    assert r.stdout.count("ok ") == 8, r.stdout
