"""Failure detection on the GPU without a fault: the kernels' bounded waits
give up, report OCCAM_ERR_TIMEOUT through the status word, and leave the
context usable (a prune call afterwards still matches the oracle)."""

from __future__ import annotations

import pytest
import torch

from synth import tiny_batch
from tests.gpu_helpers import check_prune, run_prune

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def test_bounded_waits_run_out_and_report():
    import paper_2605_29657_gb300 as occ

    mask, status = occ.occam_selftest_wait(20_000_000)
    assert mask == 7                                   # all three waits gave up
    assert status == occ._lib.OCCAM_ERR_TIMEOUT
    # the context is still usable
    b = tiny_batch(B=2, segs=2, P=(30, 11), R=2, M=(4, 9), H1=16, d1=64, H2=32, d2=128, hidden=64, seed=71,
                   beta1=2.0)
    gpu = run_prune(b, 0.3, 1.0)
    assert gpu["status"] == 0
    check_prune(b, gpu, 0.3, 1.0)
