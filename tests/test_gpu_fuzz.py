"""Seeded random small batches through occam_prune, each against the oracle.

Every case draws its own shapes and parameters: [CLS] or mutual Stage I with
each supported head size, 1-4 samples of 1-3 segments, 0-400 visual rows and
1-4 registers per segment, 1-300 text tokens, grouped-query Stage II keys,
lambda values from "keep everything" to "keep only the registers", the
register flag and the Stage-II route. The parity rules are those of
tests/gpu_helpers.check_prune (scores within 1e-3 relative, masks exact
outside the 1e-5 band)."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from synth import tiny_batch
from tests.gpu_helpers import check_prune, run_prune

pytestmark = pytest.mark.gpu

N_CASES = 100


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _case(i: int):
    rng = np.random.default_rng(20261202 + i)
    stage1 = "mutual" if rng.random() < 0.3 else "cls"
    d1 = int(rng.choice([64, 72, 80] if stage1 == "mutual" else [64, 72, 128]))
    B = int(rng.integers(1, 5))
    segs = 1 if stage1 == "mutual" else int(rng.integers(1, 4))
    P = tuple(int(x) for x in rng.integers(0, 401, size=B))
    R = int(rng.integers(1, 5))
    M = tuple(int(x) for x in rng.integers(1, 301, size=B))
    kw = dict(B=B, segs=segs, P=P, R=R, M=M, H1=16, d1=d1, H2=32, d2=128, hidden=64,
              H2kv=int(rng.choice([0, 0, 8])), stage1=stage1, seed=1000 + i, beta1=2.0,
              sinks=("count", 1), query_bias=0.5)
    lam1 = float(rng.choice([0.0, 0.05, 0.3, 1.0, 3.0]))
    lam2 = float(rng.choice([0.0, 0.5, 1.1, 2.0]))
    keep_registers = bool(rng.random() < 0.8)
    path = str(rng.choice(["auto", "narrow", "twopass"]))
    return kw, lam1, lam2, keep_registers, path


@pytest.mark.parametrize("i", range(N_CASES))
def test_random_batch_matches_oracle(i):
    kw, lam1, lam2, keep_registers, path = _case(i)
    b = tiny_batch(**kw)
    gpu = run_prune(b, lam1, lam2, keep_registers=keep_registers, path=path)
    assert gpu["status"] == 0, (kw, lam1, lam2, path)
    check_prune(b, gpu, lam1, lam2, keep_registers=keep_registers)
