"""Input generator structure and the bench's host-side logic (CPU only)."""

from __future__ import annotations

import os
import sys

import numpy as np
import pytest
import torch

from synth import make_batch, tiny_batch


def test_generator_is_deterministic_and_structured():
    a = tiny_batch(B=2, segs=2, P=(6, 9), R=2, M=(3, 4), seed=5)
    b = tiny_batch(B=2, segs=2, P=(6, 9), R=2, M=(3, 4), seed=5)
    for k in ("K1", "K2", "Q_text", "hidden"):
        assert torch.equal(a[k], b[k])
    m = a["meta"]
    assert m["seg_off_host"].tolist() == [0, 8, 16, 27, 38]
    assert m["reg_idx_host"].tolist() == [6, 7, 14, 15, 25, 26, 36, 37]   # registers end each segment
    assert m["row_off_host"].tolist() == [0, 16, 38]


def test_sinks_are_scaled_keys():
    b = tiny_batch(B=1, segs=1, P=(200,), R=1, M=(2,), sinks=("count", 5), seed=3, H1=4, d1=16, H2=2, d2=16)
    s = b["meta"]["sinks"]
    nrm = b["K1"].float().norm(dim=(1, 2))
    assert len(s) == 5 and (nrm[s].min() > 3 * nrm.median())


def test_bench_aggregate_gloo_two_ranks(tmp_path):
    import torch.multiprocessing as mp
    port = 29500 + (os.getpid() % 1000)
    mp.spawn(_agg_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True)
    got = [open(os.path.join(tmp_path, f"r{r}")).read().split() for r in range(2)]
    for ms, n in got:
        assert float(ms) == 7.5 and int(n) == 64 + 65


def _agg_worker(rank, world, port, out):
    import torch.distributed as dist
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, n = bench.aggregate([5.0, 7.5][rank], [64, 65][rank])
    with open(os.path.join(out, f"r{rank}"), "w") as f:
        f.write(f"{ms} {n}")
    dist.destroy_process_group()


def test_algorithmic_bytes_accounting():
    import bench
    meta = dict(total_rows=1000, S_tot=5, total_text=100, H1=16, d1=64, H2=32, d2=128, hidden=4096, stage1="cls")
    b = bench.algorithmic_bytes(meta, n1_total=200, kept_total=50)
    # K1 once, the [CLS] queries, 16 fp32 logits per row
    assert b["stage1"] == 1000 * 2048 + 5 * 2048 + 1000 * 16 * 4
    assert b["gather"] == 50 * 2 * 3 * 8192
    assert b["step"] > b["stage1"]
    # mutual mode: Q1 and K1 in each of the two passes
    mm = dict(meta, stage1="mutual", d1=72)
    bm = bench.algorithmic_bytes(mm, n1_total=200, kept_total=50)
    assert bm["stage1"] == 2 * 1000 * 2 * 16 * 72 * 2
    assert bm["step"] > 2 * 1000 * 16 * 72 * 2
