"""Test glue for the GPU parity tests: run the CUDA path through the C ABI
and compare it with the CPU oracle under the parity rule.

Parity rule (scores in fp32 on the GPU, float64 in the oracle):
* s1, ref1, s2, ref2: |gpu - oracle| <= 1e-3 |oracle| + 1e-5;
* keep masks bit-exact, except rows whose oracle score lies within 1e-5
  (relative) of their threshold, which are reported; when the Stage-I mask
  differs only at such rows, Stage II of the oracle is re-run on the GPU's
  Stage-I mask (a flip changes the sample's Stage-II softmax denominators);
* out_index / counts / offsets exact, gathered rows bit-exact.
"""

from __future__ import annotations

import numpy as np
import torch

from oracle import occam_oracle as O

RTOL, ATOL = 1e-3, 1e-5


def to_device(batch: dict, dev) -> dict:
    g = {}
    for k in ("q_cls", "k_cls", "Q1", "K1", "Q_text", "K_text", "K2", "hidden", "V"):
        if k in batch:
            g[k] = batch[k].to(dev).contiguous()
    return g


def run_prune(batch: dict, lam1: float, lam2: float, keep_registers: bool = True, dev="cuda",
              capacity_rows=None, gather=True, text_keys: bool = True, g=None, path: str = "auto",
              host_inputs: bool = False, rule: str = "register", budget=None, near: bool = False,
              near_rel: float = 0.0):
    """path: "auto" (fused tensor-core Stage II where it fits, wider clusters
    for small batches), "narrow" (the same without the widening) or "twopass".
    host_inputs: K2, hidden and V stay in pinned host memory (occam_prune_staged).
    rule / budget: the selection rule ("register", "mean", "budget") and the
    per-sample budget array (host ints) of the "budget" rule. near: also
    return the near-threshold flags near1 / near2 (band near_rel, 0: 1e-5)."""
    import paper_2605_29657_gb300 as occ
    route = {"auto": occ.OCCAM_ROUTE_AUTO, "twopass": occ.OCCAM_ROUTE_TWOPASS, "narrow": occ.OCCAM_ROUTE_NARROW}[path]
    old = occ.occam_set_stage2_route(route)
    try:
        return _run_prune(batch, lam1, lam2, keep_registers, dev, capacity_rows, gather, text_keys, g, host_inputs,
                          rule, budget, near, near_rel)
    finally:
        occ.occam_set_stage2_route(old)


def _run_prune(batch, lam1, lam2, keep_registers, dev, capacity_rows, gather, text_keys, g, host_inputs=False,
               rule="register", budget=None, near=False, near_rel=0.0):
    import paper_2605_29657_gb300 as occ

    m = batch["meta"]
    g = to_device(batch, dev) if g is None else g
    if host_inputs:
        g = dict(g)
        for k in ("K2", "hidden", "V"):
            g[k] = g[k].cpu().pin_memory()
    layout = occ.BatchLayout.from_batch(batch, dev)
    if m["stage1"] == "cls":
        st1 = dict(mode="cls", q=g["q_cls"], k_cls=g.get("k_cls"), K1=g["K1"])
    else:
        st1 = dict(mode="mutual", q=g["Q1"], K1=g["K1"])
    st2 = dict(Q_text=g["Q_text"], K_text=g["K_text"] if text_keys else None, K2=g["K2"])
    tensors = ()
    if gather:
        tensors = (g["hidden"], g["K2"].view(g["K2"].shape[0], -1), g["V"])
    bud = None if budget is None else torch.as_tensor(np.asarray(budget, np.int32)).to(dev)
    want = occ.PruneCall.OPTIONAL + (occ.PruneCall.NEAR if near else ())
    out = occ.occam_prune(layout, st1, st2, lam1, lam2, keep_registers=keep_registers, gather=tensors,
                          capacity_rows=capacity_rows, host_inputs=host_inputs, rule=rule, budget=bud, want=want,
                          near_rel=near_rel)
    torch.cuda.synchronize()
    status = occ.occam_get_status(out["ws"])
    res = {k: v.cpu().numpy() for k, v in out.items() if isinstance(v, torch.Tensor) and k != "ws"}
    res["gathered"] = [t.cpu() for t in out["gathered"]]
    res["status"] = status
    return res


def close(name, got, want, rtol=RTOL, atol=ATOL):
    got = np.asarray(got, np.float64)
    want = np.asarray(want, np.float64)
    err = np.abs(got - want)
    bad = err > rtol * np.abs(want) + atol
    if bad.any():
        i = int(np.argmax(err - (rtol * np.abs(want) + atol)))
        raise AssertionError(f"{name}: {int(bad.sum())} values out of tolerance; worst at {i}: "
                             f"gpu={got[i]!r} oracle={want[i]!r}")


def check_prune(batch: dict, gpu: dict, lam1: float, lam2: float, keep_registers: bool = True,
                text_keys: str = "causal", gather=True, capacity_rows=None, rule: str = "register",
                budget=None) -> dict:
    """Compares a GPU prune result with the oracle; returns a small report.

    Under the "budget" rule the Stage-II selection is an integer decision
    taken from fp32 scores: the GPU's keep2 must equal the oracle's
    budget_keep applied to the GPU's own s2 exactly, and where it differs
    from the oracle's keep2 the row's oracle s2 must lie within 1e-5
    (relative) of its sample's budget-th largest score."""
    ref = O.prune(batch, lam1, lam2, keep_registers=keep_registers, text_keys=text_keys,
                  gather=("hidden", "K2", "V") if gather else (), rule=rule, budget=budget)
    meta = batch["meta"]
    row_off = meta["row_off_host"]
    B = meta["B"]
    is_reg = ref["is_reg"]
    rep = dict(band1=0, band2=0, cascade=False)
    close("s1", gpu["s1"], ref["s1"])
    close("ref1", gpu["ref1"], ref["ref1"])
    k1 = gpu["keep1"].astype(bool)
    d1 = k1 != ref["keep1"]
    assert not (d1 & ~ref["near1"]).any(), f"keep1 differs outside the band at rows {np.nonzero(d1 & ~ref['near1'])[0][:10]}"
    assert k1[is_reg].all(), "a register row is missing from S1"
    rep["band1"] = int(d1.sum())
    if d1.any():
        rep["cascade"] = True
        ref = O.prune(batch, lam1, lam2, keep_registers=keep_registers, text_keys=text_keys,
                      keep1_override=k1, gather=("hidden", "K2", "V") if gather else (), rule=rule,
                      budget=budget)
    close("s2", gpu["s2"], ref["s2"])
    close("ref2", gpu["ref2"], ref["ref2"])
    k2 = gpu["keep2"].astype(bool)
    d2 = k2 != ref["keep2"]
    if rule == "budget":
        own, _ = O.budget_keep(gpu["s2"].astype(np.float64), row_off, k1, budget, is_reg,
                               keep_registers=keep_registers)
        assert np.array_equal(k2, own), "keep2 is not the budget selection of the GPU's own s2"
        near = np.zeros_like(d2)
        for b in range(B):
            a, z = row_off[b], row_off[b + 1]
            c = np.nonzero(k1[a:z] & ~is_reg[a:z])[0] + a
            k = min(max(int(budget[b]), 0), len(c))
            if 0 < k < len(c):
                kth = np.sort(ref["s2"][c])[::-1][k - 1]
                near[c] = np.abs(ref["s2"][c] - kth) <= 1e-5 * kth
        assert not (d2 & ~near).any(), f"keep2 differs away from the budget boundary at {np.nonzero(d2 & ~near)[0][:10]}"
    else:
        assert not (d2 & ~ref["near2"]).any(), f"keep2 differs outside the band at rows {np.nonzero(d2 & ~ref['near2'])[0][:10]}"
    rep["band2"] = int(d2.sum())
    assert (k2[is_reg] == keep_registers).all(), "register rows in keep2 must equal keep_registers"
    # compaction must be exact for the GPU's own mask
    tensors = []
    if gather:
        for name in ("hidden", "K2", "V"):
            t = batch[name].reshape(batch[name].shape[0], -1).contiguous().view(torch.int16).numpy()
            tensors.append(t)
    out_index, count_out, out_off, gathered = O.compact(k2, row_off, tensors)
    n = int(out_off[-1])
    assert gpu["out_off"].tolist() == out_off.tolist(), "out_off"
    assert gpu["count_out"].tolist() == count_out.tolist(), "count_out"
    cap = meta["total_rows"] if capacity_rows is None else capacity_rows
    m = min(n, cap)
    assert gpu["out_index"][:m].tolist() == out_index[:m].tolist(), "out_index"
    cv = [int((k2 & ~is_reg)[row_off[b]:row_off[b + 1]].sum()) for b in range(B)]
    assert gpu["count_vis"].tolist() == cv, "count_vis"
    n1 = [int((k1 & ~is_reg)[row_off[b]:row_off[b + 1]].sum()) for b in range(B)]
    assert gpu["n1_vis"].tolist() == n1, "n1_vis"
    for t, (name, want) in enumerate(zip(("hidden", "K2", "V"), gathered)):
        got = gpu["gathered"][t][:m].reshape(m, -1).contiguous().view(torch.int16).numpy()
        assert (got == want[:m]).all(), f"gathered {name} rows differ"
    if rep["band1"] == 0 and rep["band2"] == 0:
        assert gpu["count_vis"].tolist() == ref["count_vis"].tolist()
        assert gpu["out_index"][:m].tolist() == ref["out_index"][:m].tolist()
    rep["kept"] = n
    return rep
