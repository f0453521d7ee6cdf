"""Host-side checks that need no GPU: the library builds, loads, exports
every entry point include/occam.h declares, and its host validation works."""

from __future__ import annotations

import ctypes
import os
import re
import shutil

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2605_29657_gb300 import build
    build.build()
    import paper_2605_29657_gb300 as occ
    return occ.library()


def declared_functions():
    txt = open(os.path.join(ROOT, "include", "occam.h")).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(occam_\w+)\s*\(", txt, re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("occam_score_stage1", "occam_threshold", "occam_score_stage2", "occam_compact",
                 "occam_prune", "occam_workspace_size", "occam_get_status"):
        assert want in names


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def _host_batch(B=2, S=4, rows=40, text=10):
    import paper_2605_29657_gb300 as occ
    fake = 0x1000
    return occ._lib.CBatch(B, S, rows, text, 10, 20, 7, 2, fake, fake, fake, fake, fake, fake, fake)


def test_workspace_size_host_only(lib):
    import paper_2605_29657_gb300 as occ
    n = ctypes.c_size_t(0)
    b = _host_batch()
    assert lib.occam_workspace_size(ctypes.byref(b), 16, 32, ctypes.byref(n)) == 0
    small = n.value
    assert small > 0 and small % 256 == 0
    b2 = _host_batch(rows=4000)
    assert lib.occam_workspace_size(ctypes.byref(b2), 16, 32, ctypes.byref(n)) == 0
    assert n.value > small
    bad = _host_batch(B=0)
    assert lib.occam_workspace_size(ctypes.byref(bad), 16, 32, ctypes.byref(n)) == occ._lib.OCCAM_ERR_INVALID_ARG


def test_invalid_arguments_rejected_on_host(lib):
    import paper_2605_29657_gb300 as occ
    assert lib.occam_prune(None, None, None, 0, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    a = occ._lib.CPruneArgs()
    a.batch = _host_batch()
    a.stage1 = occ._lib.CStage1(0, 16, 48, 0x1000, None, 0x1000)   # d1 = 48 is not built
    a.stage2 = occ._lib.CStage2(32, 128, 0x1000, 0x1000, 0x1000)
    o = occ._lib.CPruneOut()
    assert lib.occam_prune(ctypes.byref(a), ctypes.byref(o), None, 0, None) != 0
    a.stage1 = occ._lib.CStage1(0, 16, 64, 0x1001, None, 0x1000)   # misaligned q
    assert lib.occam_prune(ctypes.byref(a), ctypes.byref(o), None, 0, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    assert lib.occam_get_status(None, None, None) == occ._lib.OCCAM_ERR_INVALID_ARG


def test_layout_validation_host_only():
    import paper_2605_29657_gb300 as occ
    ok = occ.BatchLayout([0, 10, 25], [0, 4, 10, 25], [2, 3, 9, 24], [0, 2, 3, 4], [0, 3, 5], device="cpu")
    assert ok.B == 2 and ok.S_tot == 3 and ok.max_seg_rows == 15 and ok.max_sample_rows == 15
    assert ok.host["seg_first"].tolist() == [0, 2, 3]
    assert ok.host["seg_sample"].tolist() == [0, 0, 1]
    with pytest.raises(occ.OccamError):   # a sample without text
        occ.BatchLayout([0, 10, 25], [0, 10, 25], [9, 24], [0, 1, 2], [0, 3, 3], device="cpu")
    with pytest.raises(occ.OccamError):   # a segment without registers
        occ.BatchLayout([0, 10, 25], [0, 10, 25], [9], [0, 1, 1], [0, 3, 5], device="cpu")
    with pytest.raises(occ.OccamError):   # segments that do not tile the samples
        occ.BatchLayout([0, 10, 25], [0, 12, 25], [9, 24], [0, 1, 2], [0, 3, 5], device="cpu")


def test_no_cpu_fallback_without_device():
    import torch
    import paper_2605_29657_gb300 as occ
    if torch.cuda.is_available():
        pytest.skip("has a GPU")
    lay = occ.BatchLayout([0, 10], [0, 10], [9], [0, 1], [0, 3], device="cpu")
    x = torch.zeros(10, 16, 64, dtype=torch.bfloat16)
    with pytest.raises(occ.OccamError):
        occ.occam_score_stage1(lay, occ.OCCAM_STAGE1_CLS, x[:1], x)


def test_rule_argument_checked_on_host(lib):
    import paper_2605_29657_gb300 as occ
    a = occ._lib.CPruneArgs()
    a.batch = _host_batch()
    a.stage1 = occ._lib.CStage1(0, 16, 64, 0x1000, None, 0x1000)
    a.stage2 = occ._lib.CStage2(32, 128, 0x1000, 0x1000, 0x1000)
    a.capacity_rows = 0
    o = occ._lib.CPruneOut()
    o.keep2 = o.count_vis = o.count_out = o.out_off = 0x1000
    a.rule = 7
    assert lib.occam_prune(ctypes.byref(a), ctypes.byref(o), None, 0, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    a.rule = occ.OCCAM_RULE_BUDGET                               # a budget rule needs the budget array
    assert lib.occam_prune(ctypes.byref(a), ctypes.byref(o), None, 0, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    a.rule = occ.OCCAM_RULE_MEAN                                 # valid: fails later, on the workspace
    assert lib.occam_prune(ctypes.byref(a), ctypes.byref(o), None, 0, None) == occ._lib.OCCAM_ERR_WORKSPACE


def test_selftest_arguments_checked_on_host(lib):
    import paper_2605_29657_gb300 as occ
    assert lib.occam_selftest_wait(0, None, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    assert lib.occam_selftest_wait(10 ** 6, None, None) == occ._lib.OCCAM_ERR_INVALID_ARG
    assert lib.occam_selftest_wait(2 * 10 ** 9, 0x1000, None) == occ._lib.OCCAM_ERR_INVALID_ARG


def test_ctypes_structs_match_the_header(tmp_path):
    """The binding's ctypes structs have the header's layout: a C program
    compiled against include/occam.h prints every field's offset and each
    struct's size, and ctypes must agree (an ABI drift between the two would
    pass wrong pointers silently)."""
    import shutil
    import subprocess

    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no C compiler")
    occ = pytest.importorskip("paper_2605_29657_gb300")
    L = occ._lib
    structs = {"occam_batch": L.CBatch, "occam_stage1_args": L.CStage1, "occam_stage2_args": L.CStage2,
               "occam_prune_args": L.CPruneArgs, "occam_prune_out": L.CPruneOut}
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "occam.h"', "int main(void) {"]
    for cname, py in structs.items():
        lines.append(f'  printf("{cname} size %zu\\n", sizeof({cname}));')
        for fname, _ in py._fields_:
            lines.append(f'  printf("{cname}.{fname} %zu\\n", offsetof({cname}, {fname}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "layout"
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    subprocess.run([cc, "-std=c11", "-I", os.path.join(root, "include"), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], check=True, capture_output=True, text=True).stdout.split("\n")
    got = dict(line.rsplit(" ", 1) for line in out if line)
    for cname, py in structs.items():
        assert int(got[f"{cname} size"]) == ctypes.sizeof(py), cname
        for fname, _ in py._fields_:
            assert int(got[f"{cname}.{fname}"]) == getattr(py, fname).offset, f"{cname}.{fname}"
