"""Calibrate the synthetic workloads' free parameters with the CPU oracle.

The paper fixes lambda1 for LLaVA-v1.5 / LLaVA-NeXT (App. A "Parameter
settings"; Table 5) and picks lambda2 by budget matching (App. A, Eq. 19:
lambda2* = argmin |mean |S2|(lambda2) - K_tar|, from a calibration set). This
script does the same on each seeded synthetic batch:

1. beta1 (the register key's logit gain) is bisected so that the mean Stage-I
   survivor count matches the paper's N1 (Table 5: 523 of 2,880 on LLaVA-NeXT
   at lambda1 = 0.045; App. A: "about 200--300" on LLaVA-v1.5, 250 used here).
   For the mutual-scoring workload the paper gives no lambda1, so beta1 is
   fixed and lambda1 is matched to the target instead;
2. lambda2 is matched exactly to the final budget (Eq. 19): the count is a
   step function of lambda2, so lambda2 is placed between the ratios
   s2(v)/s2(r) that bracket the target total.

Only ``synth`` (inputs) and ``oracle`` (the CPU definition) are used. Output:
``synth/calibrated.json``. Run: ``python -m synth.calibrate [names...]``.
"""

from __future__ import annotations

import json
import os
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, os.path.dirname(_HERE))

from oracle import occam_oracle as O  # noqa: E402
from synth.configs import WORKLOADS, get_config  # noqa: E402
from synth.gen import make_batch  # noqa: E402


def _stage1(batch):
    m = batch["meta"]
    if m["stage1"] == "cls":
        return O.stage1_cls(batch["q_cls"], batch["k_cls"], batch["K1"], m["seg_off_host"],
                            m["reg_idx_host"], m["reg_off_host"])
    return O.stage1_mutual(batch["Q1"], batch["K1"], m["seg_off_host"], m["reg_idx_host"],
                           m["reg_off_host"])


def _ratios1(batch):
    """Per visual row: s1(v) / s1(r) of its segment."""
    m = batch["meta"]
    s1, ref1 = _stage1(batch)
    seg_of_row = np.repeat(np.arange(m["S_tot"]), np.diff(m["seg_off_host"]))
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    return s1 / ref1[seg_of_row], is_reg


def _n1_target(w, P):
    t = w.targets
    return t["n1_vis"] if "n1_vis" in t else t["n1_frac"] * float(np.mean(P)) * w.segs


def _count_target(w, P):
    t = w.targets
    return t["count_vis"] if "count_vis" in t else t["count_frac"] * float(np.mean(P)) * w.segs


def _match(ratios_desc: np.ndarray, total_target: float) -> float:
    """lambda placed halfway (geometrically) between the ratios around the target count."""
    k = int(round(total_target))
    k = max(1, min(k, len(ratios_desc) - 1))
    return float(np.sqrt(ratios_desc[k - 1] * ratios_desc[k]))


def calibrate(name: str) -> dict:
    w = get_config(name)
    res = {}
    if w.stage1 == "cls":
        lo, hi = 0.0, 12.0
        for _ in range(22):
            beta = 0.5 * (lo + hi)
            b = make_batch(get_config(name, beta1=beta), with_stage2=False, with_gather=False)
            r, is_reg = _ratios1(b)
            n1 = float(np.sum((r >= w.lambda1) & ~is_reg)) / w.B
            if n1 > _n1_target(w, b["meta"]["P"]):
                lo = beta
            else:
                hi = beta
        res["beta1"] = round(0.5 * (lo + hi), 5)
        res["lambda1"] = w.lambda1
    else:
        beta = w.beta1
        b = make_batch(get_config(name, beta1=beta), with_stage2=False, with_gather=False)
        r, is_reg = _ratios1(b)
        vis = np.sort(r[~is_reg])[::-1]
        res["beta1"] = beta
        res["lambda1"] = round(_match(vis, _n1_target(w, b["meta"]["P"]) * w.B), 6)
    w2 = get_config(name, beta1=res["beta1"], lambda1=res["lambda1"])
    b = make_batch(w2, with_gather=False)
    m = b["meta"]
    out = O.prune(b, w2.lambda1, 1.0, gather=())
    sample_of_row = np.repeat(np.arange(m["B"]), np.diff(m["row_off_host"]))
    cand = out["keep1"] & ~out["is_reg"]
    ratios = np.sort((out["s2"] / out["ref2"][sample_of_row])[cand])[::-1]
    res["lambda2"] = round(_match(ratios, _count_target(w, m["P"]) * m["B"]), 6)
    fin = O.prune(b, w2.lambda1, res["lambda2"], gather=())
    res["mean_n1_vis"] = float(np.mean(fin["n1_vis"]))
    res["mean_count_vis"] = float(np.mean(fin["count_vis"]))
    return res


def main(argv):
    names = argv[1:] or WORKLOADS
    path = os.path.join(_HERE, "calibrated.json")
    cal = json.load(open(path)) if os.path.exists(path) else {}
    for n in names:
        cal[n] = calibrate(n)
        print(n, cal[n], flush=True)
        with open(path, "w") as f:
            json.dump(cal, f, indent=1, sort_keys=True)


if __name__ == "__main__":
    main(sys.argv)
