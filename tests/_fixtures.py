"""Test glue: turn the hand-derived worked example into a batch dict."""

from __future__ import annotations

import json
import os

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))


def worked_example() -> tuple[dict, dict]:
    with open(os.path.join(HERE, "golden", "worked_example.json")) as f:
        g = json.load(f)
    bf = lambda k: torch.tensor(g[k], dtype=torch.float32).to(torch.bfloat16)  # noqa: E731
    batch = {k: bf(k) for k in ("q_cls", "k_cls", "K1", "Q_text", "K_text", "K2")}
    lay = dict(
        row_off=np.array([0, 4], np.int64), seg_off=np.array([0, 4], np.int64),
        seg_sample=np.array([0], np.int32), reg_idx=np.array([3], np.int32),
        reg_off=np.array([0, 1], np.int32), text_off=np.array([0, 2], np.int64),
    )
    for k, v in lay.items():
        batch[k] = torch.as_tensor(v)
    batch["hidden"] = torch.arange(4 * 8, dtype=torch.float32).reshape(4, 8).to(torch.bfloat16)
    batch["V"] = (-torch.arange(4 * 8, dtype=torch.float32)).reshape(4, 8).to(torch.bfloat16)
    batch["meta"] = dict(
        name="worked_example", B=1, S_tot=1, total_rows=4, total_text=2, max_seg_rows=4,
        max_sample_rows=4, max_text=2, min_text=2, regs_per_seg=1, segs_per_sample=1,
        H1=1, d1=4, H2=1, d2=4, hidden=8, stage1="cls", P=np.array([3]), M=np.array([2]),
        **{k + "_host": v for k, v in lay.items()},
    )
    return batch, g
