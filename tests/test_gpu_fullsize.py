"""Full-size workloads in the bench's launch configuration, checked on
sampled samples against the oracle (samples are independent, so a sample's
outputs can be recomputed alone) and on properties that hold at any size."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import batch_slice_to_host, get_config, make_batch
from tests.gpu_helpers import check_prune, run_prune

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _global_properties(batch, gpu):
    m = batch["meta"]
    B, R = m["B"], m["total_rows"]
    out_off = gpu["out_off"]
    assert out_off[0] == 0 and (np.diff(out_off) >= 0).all()
    assert np.array_equal(np.diff(out_off), gpu["count_out"])
    n = int(out_off[-1])
    assert n == int(gpu["keep2"].astype(bool).sum())
    idx = gpu["out_index"][:n]
    assert (np.diff(idx) > 0).all() and idx[0] >= 0 and idx[-1] < R
    assert gpu["keep2"][idx].all()
    assert (gpu["count_vis"] <= gpu["n1_vis"]).all()


def _slice_gpu(gpu, batch, samples):
    """The chosen samples' part of a full-batch GPU result, re-based like batch_slice_to_host."""
    m = batch["meta"]
    ro = m["row_off_host"]
    rows = np.concatenate([np.arange(ro[b], ro[b + 1]) for b in samples])
    segs = np.concatenate([np.arange(b * m["segs_per_sample"], (b + 1) * m["segs_per_sample"]) for b in samples])
    out = {k: gpu[k][rows] for k in ("s1", "s2", "keep1", "keep2")}
    out["ref1"] = gpu["ref1"][segs]
    for k in ("ref2", "count_vis", "count_out", "n1_vis"):
        out[k] = gpu[k][samples]
    idx, offs, gath = [], [0], [[], [], []]
    base = 0
    for b in samples:
        a, z = int(gpu["out_off"][b]), int(gpu["out_off"][b + 1])
        idx.append(gpu["out_index"][a:z] - ro[b] + base)
        for t in range(3):
            gath[t].append(gpu["gathered"][t][a:z])
        offs.append(offs[-1] + (z - a))
        base += ro[b + 1] - ro[b]
    out["out_index"] = np.concatenate(idx)
    out["out_off"] = np.asarray(offs)
    out["gathered"] = [torch.cat(g) for g in gath]
    return out


@pytest.mark.parametrize("name,samples", [
    ("llavanext_b64", [0, 21, 42, 63]),
    ("video_b4", [0, 1, 2, 3]),
    ("qwen3vl_b32", None),
])
def test_fullsize_sampled(name, samples):
    w = get_config(name)
    batch = make_batch(w, device="cuda")
    gpu = run_prune(batch, w.lambda1, w.lambda2)
    assert gpu["status"] == 0
    _global_properties(batch, gpu)
    if samples is None:  # the smallest, the largest and one in between
        P = np.asarray(batch["meta"]["P"])
        order = np.argsort(P)
        samples = sorted({int(order[0]), int(order[len(P) // 2]), int(order[-1])})
    host = batch_slice_to_host(batch, samples)
    sub = _slice_gpu(gpu, batch, samples)
    rep = check_prune(host, sub, w.lambda1, w.lambda2)
    print(name, samples, rep, "mean n1", gpu["n1_vis"].mean(), "mean count", gpu["count_vis"].mean())
