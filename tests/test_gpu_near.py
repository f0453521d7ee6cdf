"""Near-threshold flags of occam_prune: the rows whose keep decision in the
Stage-I test (Eq. 5) or the Stage-II test (Eq. 8) turns on the last digits of
their score, |s - tau| <= near_rel * |tau|."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import occam_oracle as O
from synth import tiny_batch
from tests.gpu_helpers import run_prune

pytestmark = pytest.mark.gpu

H = dict(H1=16, d1=64, H2=32, d2=128)
F = np.float32


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _tiny(**kw):
    args = dict(H, hidden=256, beta1=2.0, sinks=("count", 1))
    args.update(kw)
    return tiny_batch(**args)


def _replica(b, gpu, lam1, lam2, rel):
    """The device's near test in fp32 from the GPU's own scores and references:
    tau = fl(lambda * ref), then |s - tau| <= rel * |tau| (visual rows; S1
    rows only for Stage II)."""
    m = b["meta"]
    seg = np.repeat(np.arange(m["S_tot"]), np.diff(m["seg_off_host"]))
    samp = np.repeat(np.arange(m["B"]), np.diff(m["row_off_host"]))
    reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    tau1 = (F(lam1) * gpu["ref1"].astype(F)).astype(F)[seg]
    tau2 = (F(lam2) * gpu["ref2"].astype(F)).astype(F)[samp]
    s1, s2 = gpu["s1"].astype(F), gpu["s2"].astype(F)
    near1 = ~reg & (np.abs(s1 - tau1) <= F(rel) * np.abs(tau1))
    near2 = ~reg & (gpu["keep1"] != 0) & (np.abs(s2 - tau2) <= F(rel) * np.abs(tau2))
    return near1, near2


@pytest.mark.parametrize("stage1", ["cls", "mutual"])
def test_near_flags_mark_rows_on_the_threshold(stage1):
    kw = dict(B=3, segs=2, P=(200, 90, 300), R=4, M=(64, 129, 20), seed=41)
    if stage1 == "mutual":
        kw.update(segs=1, stage1="mutual", d1=72, query_bias=0.5)
    b = _tiny(**kw)
    m = b["meta"]
    reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    seg = np.repeat(np.arange(m["S_tot"]), np.diff(m["seg_off_host"]))
    samp = np.repeat(np.arange(m["B"]), np.diff(m["row_off_host"]))
    # lambda1 that puts a mid-ranked visual row of segment 0 on its threshold
    a = run_prune(b, 0.3, 1.2, gather=False)
    vis0 = np.flatnonzero(~reg & (seg == 0))
    r0 = int(vis0[np.argsort(a["s1"][vis0])[len(vis0) // 2]])
    lam1 = float(F(a["s1"][r0]) / F(a["ref1"][seg[r0]]))
    # lambda2 that puts a visual S1 row of sample 0 on its threshold (s2 does
    # not depend on lambda2, so the last call sees the same scores)
    c = run_prune(b, lam1, 1.2, gather=False)
    s1rows = np.flatnonzero(~reg & (c["keep1"] != 0) & (samp == 0))
    assert len(s1rows) > 0
    r1 = int(s1rows[np.argsort(c["s2"][s1rows])[len(s1rows) // 2]])
    lam2 = float(F(c["s2"][r1]) / F(c["ref2"][0]))
    gpu = run_prune(b, lam1, lam2, gather=False, near=True)
    assert gpu["status"] == 0
    assert np.array_equal(gpu["s2"], c["s2"])
    want1, want2 = _replica(b, gpu, lam1, lam2, 1e-5)
    assert np.array_equal(gpu["near1"] != 0, want1)
    assert np.array_equal(gpu["near2"] != 0, want2)
    assert gpu["near1"][r0] == 1 and gpu["near2"][r1] == 1
    # registers are never flagged
    assert not gpu["near1"][reg].any() and not gpu["near2"][reg].any()


def test_near_band_argument():
    b = _tiny(B=2, segs=2, P=(120, 57), R=3, M=(30, 5), seed=42)
    for rel in (0.5, 0.05):
        gpu = run_prune(b, 0.3, 1.1, gather=False, near=True, near_rel=rel)
        want1, want2 = _replica(b, gpu, 0.3, 1.1, rel)
        assert np.array_equal(gpu["near1"] != 0, want1), rel
        assert np.array_equal(gpu["near2"] != 0, want2), rel
        assert want1.any()  # a band this wide holds rows


def test_near2_is_empty_under_the_budget_rule():
    b = _tiny(B=2, segs=1, P=(90, 140), R=2, M=(12, 40), seed=43)
    gpu = run_prune(b, 0.2, 1.0, gather=False, near=True, near_rel=0.5, rule="budget", budget=[10, 20])
    assert gpu["status"] == 0
    assert not gpu["near2"].any()
    want1, _ = _replica(b, gpu, 0.2, 1.0, 0.5)
    assert np.array_equal(gpu["near1"] != 0, want1)
