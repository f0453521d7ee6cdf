"""Properties of the threshold rule that hold exactly on the device's own
results, at full size (the LLaVA-NeXT-shaped batch of 8), without the oracle:

* the scores of a stage do not depend on its lambda, and the fp32 product
  lambda * ref grows with lambda, so the kept sets of the image-adaptive test
  (Eq. 5) shrink as lambda1 grows, and those of the query-adaptive test
  (Eq. 8) shrink as lambda2 grows with lambda1 fixed: the masks are nested;
* registers are in S1 and follow keep_registers in the output, never as
  candidates;
* the compacted list is ascending within each sample, sample-major, and the
  offsets are the prefix sums of the counts."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import get_config, make_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


@pytest.fixture(scope="module")
def nextb8():
    import paper_2605_29657_gb300 as occ
    w = get_config("llavanext_b8")
    b = make_batch(w, "cuda", with_gather=False)
    layout = occ.BatchLayout.from_batch(b, "cuda")

    def run(lam1, lam2, keep_registers=True):
        out = occ.occam_prune(layout, dict(mode="cls", q=b["q_cls"], k_cls=b["k_cls"], K1=b["K1"]),
                              dict(Q_text=b["Q_text"], K_text=b["K_text"], K2=b["K2"]), lam1, lam2,
                              keep_registers=keep_registers, want=occ.PruneCall.OPTIONAL)
        torch.cuda.synchronize()
        assert occ.occam_get_status(out["ws"]) == 0
        return {k: v.cpu().numpy() for k, v in out.items() if isinstance(v, torch.Tensor) and k != "ws"}

    meta = b["meta"]
    reg = np.zeros(meta["total_rows"], bool)
    reg[np.asarray(meta["reg_idx_host"])] = True
    return w, run, meta, reg


def test_stage2_masks_nest_in_lambda2(nextb8):
    w, run, meta, reg = nextb8
    prev = None
    for lam2 in (0.0, 0.5 * w.lambda2, w.lambda2, 1.5 * w.lambda2, 4.0 * w.lambda2):
        r = run(w.lambda1, lam2)
        k2 = r["keep2"].astype(bool)
        if prev is not None:
            assert np.array_equal(r["s2"], prev["s2"]), "s2 depends on lambda2"
            assert not (k2 & ~prev["keep2"].astype(bool)).any(), "a row kept at a larger lambda2 was dropped at a smaller one"
            assert (r["count_vis"] <= prev["count_vis"]).all()
        assert k2[reg].all() and not (k2 & ~r["keep1"].astype(bool)).any()
        prev = r


def test_stage1_masks_nest_in_lambda1(nextb8):
    w, run, meta, reg = nextb8
    prev = None
    for lam1 in (0.0, 0.5 * w.lambda1, w.lambda1, 2.0 * w.lambda1, 8.0 * w.lambda1):
        r = run(lam1, w.lambda2)
        k1 = r["keep1"].astype(bool)
        if prev is not None:
            assert np.array_equal(r["s1"], prev["s1"]), "s1 depends on lambda1"
            assert not (k1 & ~prev["keep1"].astype(bool)).any(), "a row in S1 at a larger lambda1 left it at a smaller one"
            assert (r["n1_vis"] <= prev["n1_vis"]).all()
        assert k1[reg].all(), "registers are always in S1"
        prev = r


@pytest.mark.parametrize("keep_registers", [True, False])
def test_compacted_list_order_and_offsets(nextb8, keep_registers):
    w, run, meta, reg = nextb8
    r = run(w.lambda1, w.lambda2, keep_registers=keep_registers)
    row_off = np.asarray(meta["row_off_host"])
    k2 = r["keep2"].astype(bool)
    assert (k2[reg] == keep_registers).all()
    off = r["out_off"]
    assert off[0] == 0 and np.array_equal(np.diff(off), r["count_out"])
    idx = r["out_index"][: off[-1]]
    for b in range(meta["B"]):
        rows = idx[off[b]:off[b + 1]]
        assert (np.diff(rows) > 0).all(), "not ascending within the sample"
        assert ((rows >= row_off[b]) & (rows < row_off[b + 1])).all(), "a row outside its sample"
        assert np.array_equal(rows, np.flatnonzero(k2[row_off[b]:row_off[b + 1]]) + row_off[b])
    assert np.array_equal(r["count_vis"], [int((k2 & ~reg)[row_off[b]:row_off[b + 1]].sum()) for b in range(meta["B"])])
