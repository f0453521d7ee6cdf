"""occam_compact_noalloc: the compaction entry point for callers that cannot
allocate device memory (it uses the library's fixed scratch array instead of
a workspace). Its output must equal the oracle's compaction and
occam_compact's on the same inputs, on two calls in a row (the second call
reuses the array the first one left behind). This file is collected last on
purpose."""

from __future__ import annotations

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


def _batch():
    from synth import tiny_batch
    # several 2,048-row scan tiles with a ragged tail
    return tiny_batch(B=4, segs=2, P=(900, 17, 1500, 640), R=3, M=(2, 3, 4, 5), H1=2, d1=8, H2=2, d2=8,
                      hidden=64, seed=31)


def test_noalloc_matches_workspace_entry_two_calls():
    import __graft_entry__ as g
    g.build()
    import paper_2605_29657_gb300 as occ
    from oracle import occam_oracle as O

    assert torch.cuda.is_available()
    b = _batch()
    dev = torch.device("cuda")
    layout = occ.BatchLayout.from_batch(b, dev)
    tensors = (b["hidden"].to(dev), b["V"].to(dev))
    rng = np.random.default_rng(5)
    R = layout.total_rows
    for call, frac in enumerate((0.3, 0.7)):
        mask = torch.tensor((rng.random(R) < frac).astype(np.uint8), device=dev)
        want = occ.occam_compact(layout, mask, tensors=tensors)
        got = occ.occam_compact_noalloc(layout, mask, tensors=tensors)
        torch.cuda.synchronize()
        n = int(want["out_off"][-1])
        assert n == int(mask.sum())
        # against the oracle's compaction of the same mask and tensors (bit-exact)
        r_index, r_count, r_off, r_rows = O.compact(mask.cpu().numpy().astype(bool), b["meta"]["row_off_host"],
                                                    tensors=[t.cpu().view(torch.int16).numpy() for t in tensors])
        assert np.array_equal(got["out_off"].cpu().numpy(), r_off), f"call {call}: oracle out_off"
        assert np.array_equal(got["count_out"].cpu().numpy(), r_count), f"call {call}: oracle counts"
        assert np.array_equal(got["out_index"][:n].cpu().numpy(), r_index), f"call {call}: oracle index"
        for t in range(len(tensors)):
            assert np.array_equal(got["gathered"][t][:n].cpu().view(torch.int16).numpy(), r_rows[t]), \
                f"call {call}: oracle gathered {t}"
        assert torch.equal(got["out_off"], want["out_off"]), f"call {call}: out_off"
        assert torch.equal(got["count_out"], want["count_out"]), f"call {call}: count_out"
        assert torch.equal(got["out_index"][:n], want["out_index"][:n]), f"call {call}: out_index"
        for t in range(len(tensors)):
            assert torch.equal(got["gathered"][t][:n].view(torch.int16),
                               want["gathered"][t][:n].view(torch.int16)), f"call {call}: gathered {t}"


def test_noalloc_rejects_batches_beyond_its_scratch():
    import paper_2605_29657_gb300 as occ
    from paper_2605_29657_gb300 import _lib as L

    lib = occ.library()
    fake = 0x1000
    big = L.CBatch(1, 1, 8192 * 2048 + 1, 1, 10, 10, 1, 1, fake, fake, fake, fake, fake, fake, fake)
    import ctypes
    rc = lib.occam_compact_noalloc(ctypes.byref(big), fake, 0, None, None, None, 0, None, fake, fake, None)
    assert rc == L.OCCAM_ERR_UNSUPPORTED
