"""Parity cases run against the bounds-checked build (liboccam_checked.so):
each must end with device status 0 (no index outside its buffer) and match
the oracle under the parity rule. Run as a script in its own process (the
binding loads one library per process); exits non-zero on any failure."""

from __future__ import annotations

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def main() -> int:
    import numpy as np
    import torch

    from paper_2605_29657_gb300 import _lib as L
    from paper_2605_29657_gb300 import build as pb

    L.use_library(pb.LIB_CHECKED)
    import paper_2605_29657_gb300 as occ
    from oracle import occam_oracle as O
    from synth import tiny_batch
    from tests.gpu_helpers import check_prune, run_prune

    assert "liboccam_checked.so" in occ.library()._name
    H = dict(H1=16, d1=64, H2=32, d2=128)

    def tiny(**kw):
        args = dict(H, hidden=256, beta1=2.0, sinks=("count", 1))
        args.update(kw)
        return tiny_batch(**args)

    cases = [
        # fused 4-CTA clusters, several text tiles and scan tiles
        ("fused4", dict(B=4, segs=2, P=(500, 333, 612, 47), R=4, M=(9, 129, 65, 2), seed=5), 0.2, 1.05, "narrow"),
        # 8-CTA clusters
        ("fused8", dict(B=2, segs=1, P=(1000, 1532), R=4, M=(130, 33), seed=25), 0.0, 1.15, "narrow"),
        # a small batch on 16-CTA clusters (widening, head split)
        ("fused16", dict(B=1, segs=1, P=(764,), R=4, M=(40,), seed=22), 0.0, 1.2, "auto"),
        # every sample on the two-pass kernels
        ("twopass", dict(B=3, segs=2, P=(5, 37, 130), R=2, M=(1, 7, 70), seed=2), 0.4, 1.1, "twopass"),
        # one sample above the fused limit (two-pass) beside a fused one
        ("mixed", dict(B=2, segs=1, P=(1700, 200), R=3, M=(70, 90), seed=23), 0.0, 1.1, "auto"),
    ]
    for name, kw, l1, l2, path in cases:
        b = tiny(**kw)
        gpu = run_prune(b, l1, l2, path=path)
        assert gpu["status"] == 0, f"{name}: status {gpu['status']}"
        check_prune(b, gpu, l1, l2)
        print("ok", name, flush=True)
    # mutual Stage I (tensor-core passes)
    b = tiny(B=3, segs=1, P=(60, 301, 150), R=4, M=(5, 90, 64), stage1="mutual", d1=72, seed=6, query_bias=0.5,
             beta1=2.0)
    gpu = run_prune(b, 0.5, 1.1)
    assert gpu["status"] == 0, f"mutual: status {gpu['status']}"
    check_prune(b, gpu, 0.5, 1.1)
    print("ok mutual", flush=True)
    # compaction alone and the no-allocation entry point, against the oracle
    b = tiny_batch(B=4, segs=2, P=(900, 17, 1500, 640), R=3, M=(2, 3, 4, 5), H1=2, d1=8, H2=2, d2=8, hidden=64,
                   seed=31)
    dev = torch.device("cuda")
    layout = occ.BatchLayout.from_batch(b, dev)
    tensors = (b["hidden"].to(dev), b["V"].to(dev))
    mask = torch.tensor((np.random.default_rng(5).random(layout.total_rows) < 0.4).astype(np.uint8), device=dev)
    r_index, r_count, r_off, r_rows = O.compact(mask.cpu().numpy().astype(bool), b["meta"]["row_off_host"],
                                                tensors=[t.cpu().view(torch.int16).numpy() for t in tensors])
    ws = occ.alloc_workspace(layout, 1, 1)
    for which in ("compact", "noalloc"):
        got = (occ.occam_compact(layout, mask, tensors=tensors, ws=ws) if which == "compact" else
               occ.occam_compact_noalloc(layout, mask, tensors=tensors))
        torch.cuda.synchronize()
        n = int(r_off[-1])
        assert np.array_equal(got["out_off"].cpu().numpy(), r_off), which
        assert np.array_equal(got["count_out"].cpu().numpy(), r_count), which
        assert np.array_equal(got["out_index"][:n].cpu().numpy(), r_index), which
        for t in range(len(tensors)):
            assert np.array_equal(got["gathered"][t][:n].cpu().view(torch.int16).numpy(), r_rows[t]), which
        print("ok", which, flush=True)
    assert occ.occam_get_status(ws) == 0, "compaction status"
    return 0


if __name__ == "__main__":
    sys.exit(main())
