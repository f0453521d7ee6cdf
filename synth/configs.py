"""Workload shapes for the five synthetic configurations.

Shapes follow the paper's settings: 576 visual tokens for LLaVA-v1.5 (Sec. 4,
Table 1), 2,880 = 5 crops x 576 for LLaVA-NeXT (Sec. 4, Table 2), Qwen3-VL with
a variable visual length and no [CLS] token (Table 3; App. A "Architecture-
specific instantiations"), and a video setting that pools the tokens of all
frames into one visual set (App. A, Eq. 20).

lambda1 follows App. A "Parameter settings": 0.01-0.02 for LLaVA-v1.5 (0.015
used here) and 0.045 (the default of Table 5) for LLaVA-NeXT-shaped inputs.
beta1 (the logit gain of the register key, which sets how much attention the
register absorbs), the Qwen lambda1 and every lambda2 are calibrated with the
CPU oracle on these synthetic inputs (``synth/calibrate.py``) to the budgets
the paper reports, and are stored in ``synth/calibrated.json``.
"""

from __future__ import annotations

import json
import os
from dataclasses import dataclass, field, replace

_HERE = os.path.dirname(os.path.abspath(__file__))


@dataclass(frozen=True)
class Workload:
    name: str
    description: str
    B: int                      # samples (images / videos) in the batch
    segs: int                   # segments per sample (crops / frames)
    vis: tuple                  # ("fixed", P) or ("uniform_step", lo, hi, step)
    regs: int                   # register rows per segment
    stage1: str                 # "cls" or "mutual"
    H1: int
    d1: int
    sinks: tuple                # ("count", n) or ("frac", f): per segment
    dup: tuple | None           # ("neighbour", frac, rho) or ("frame", frac, rho)
    M: tuple                    # ("fixed", m) or ("uniform", lo, hi)
    seed: int
    H2: int = 32
    d2: int = 128
    H2kv: int = 0               # key / value heads of K2, K_text (0: H2; fewer: grouped-query attention)
    hidden: int = 4096
    query_bias: float = 0.0     # mutual mode: per-segment shared query component (fraction of sqrt(d1))
    lambda1: float = 0.045
    lambda2: float = 1.3
    beta1: float = 4.0
    targets: dict = field(default_factory=dict)


_BASE = [
    Workload(
        name="llava15_b1",
        description="LLaVA-v1.5-shaped, batch 1: 576 visual + 4 registers, 1 CLS, 3 sinks, 32 text tokens",
        B=1, segs=1, vis=("fixed", 576), regs=4, stage1="cls", H1=16, d1=64,
        sinks=("count", 3), dup=None, M=("fixed", 32), seed=0,
        lambda1=0.015, targets={"n1_vis": 250.0, "count_vis": 64.0},
    ),
    Workload(
        name="llavanext_b8",
        description="LLaVA-NeXT-shaped, batch 8: 5 crops x (576 + 4 registers), 1% sinks, 30% near-duplicates, 64 text tokens",
        B=8, segs=5, vis=("fixed", 576), regs=4, stage1="cls", H1=16, d1=64,
        sinks=("frac", 0.01), dup=("neighbour", 0.30, 0.98), M=("fixed", 64), seed=1,
        lambda1=0.045, targets={"n1_vis": 523.0, "count_vis": 160.0},
    ),
    Workload(
        name="llavanext_b64",
        description="LLaVA-NeXT-shaped, batch 64: as llavanext_b8 with text lengths uniform in 16..256",
        B=64, segs=5, vis=("fixed", 576), regs=4, stage1="cls", H1=16, d1=64,
        sinks=("frac", 0.01), dup=("neighbour", 0.30, 0.98), M=("uniform", 16, 256), seed=2,
        lambda1=0.045, targets={"n1_vis": 523.0, "count_vis": 160.0},
    ),
    Workload(
        name="qwen3vl_b32",
        description="Qwen3-VL-shaped, ragged batch 32: 256..4096 visual tokens (step 4) + 4 registers, mutual scoring, d1=72, 1% sinks, 32..512 text tokens",
        B=32, segs=1, vis=("uniform_step", 256, 4096, 4), regs=4, stage1="mutual", H1=16, d1=72,
        sinks=("frac", 0.01), dup=None, M=("uniform", 32, 512), seed=3, query_bias=0.5,
        lambda1=0.5, beta1=3.0, targets={"n1_frac": 0.5, "count_frac": 0.222},
    ),
    Workload(
        name="qwen3vl_b16",
        description="Qwen3-VL-shaped, ragged batch 16 (the small case for kernel profiling): as qwen3vl_b32",
        B=16, segs=1, vis=("uniform_step", 256, 4096, 4), regs=4, stage1="mutual", H1=16, d1=72,
        sinks=("frac", 0.01), dup=None, M=("uniform", 32, 512), seed=5, query_bias=0.5,
        lambda1=0.5, beta1=3.0, targets={"n1_frac": 0.5, "count_frac": 0.222},
    ),
    Workload(
        name="video_b4",
        description="video-shaped, batch 4: 16 frames x (1024 + 4 registers), 50% inter-frame duplicates, 1% sinks, 128 text tokens",
        B=4, segs=16, vis=("fixed", 1024), regs=4, stage1="cls", H1=16, d1=64,
        sinks=("frac", 0.01), dup=("frame", 0.50, 0.99), M=("fixed", 128), seed=4,
        lambda1=0.045, targets={"n1_frac": 0.18, "count_frac": 0.056},
    ),
]


def _load_calibrated() -> dict:
    path = os.path.join(_HERE, "calibrated.json")
    if not os.path.exists(path):
        return {}
    with open(path) as f:
        return json.load(f)


def _apply(cal: dict) -> dict:
    out = {}
    for w in _BASE:
        c = cal.get(w.name, {})
        kw = {k: c[k] for k in ("lambda1", "lambda2", "beta1") if k in c}
        out[w.name] = replace(w, **kw)
    return out


CONFIGS: dict[str, Workload] = _apply(_load_calibrated())
WORKLOADS: list[str] = [w.name for w in _BASE]

# The throughput configuration: LLaVA-NeXT-shaped, batch 64.
HEADLINE = "llavanext_b64"


def get_config(name: str, **overrides) -> Workload:
    w = CONFIGS[name]
    return replace(w, **overrides) if overrides else w
