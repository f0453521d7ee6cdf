"""CUDA path against the CPU oracle for the rows beyond the pruning path:
n_eff of the Stage-I attention (Sec. 3.2, Observation 1)."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import occam_oracle as O
from synth import get_config, make_batch, tiny_batch
from tests.gpu_helpers import run_prune

pytestmark = pytest.mark.gpu

RTOL, ATOL = 1e-3, 1e-5


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


@pytest.mark.parametrize("case", ["tiny", "tiny_no_cls_key", "llava15_b1", "llavanext_b8"])
def test_neff_matches_oracle(case):
    if case.startswith("tiny"):
        b = tiny_batch(B=3, segs=2, P=(40, 7, 130), R=3, M=(5, 9, 2), H1=16, d1=64, H2=32, d2=128, hidden=64,
                       seed=41)
        if case == "tiny_no_cls_key":
            del b["k_cls"]
    else:
        b = make_batch(get_config(case), "cpu", with_gather=False)
    m = b["meta"]
    w = get_config(case) if not case.startswith("tiny") else None
    lam1, lam2 = (w.lambda1, w.lambda2) if w else (0.3, 1.0)
    gpu = run_prune(b, lam1, lam2, gather=False)
    assert gpu["status"] == 0
    want = O.stage1_neff(b["q_cls"], b.get("k_cls"), b["K1"], m["seg_off_host"])
    got = gpu["n_eff"].reshape(want.shape)
    np.testing.assert_allclose(got, want, rtol=RTOL, atol=ATOL)
    n_keys = np.diff(m["seg_off_host"]) + (0 if b.get("k_cls") is None else 1)
    assert (got >= 1 - 1e-4).all() and (got <= n_keys[:, None] * (1 + 1e-4)).all()


# ----------------------------------------------------------------------------- lambda2 budget matching (App. A)

def _lambda2_case(b, s2, ref2, keep1, K):
    import paper_2605_29657_gb300 as occ

    m = b["meta"]
    layout = occ.BatchLayout.from_batch(b, "cuda")
    _lambda2_check(layout, m["total_rows"], m["reg_idx_host"], m["row_off_host"], s2, ref2, keep1, K)


def _lambda2_check(layout, total_rows, reg_idx, row_off, s2, ref2, keep1, K):
    import paper_2605_29657_gb300 as occ

    lam, n = occ.occam_calibrate_lambda2(layout, torch.from_numpy(s2).cuda(), torch.from_numpy(ref2).cuda(),
                                         torch.from_numpy(keep1.astype(np.uint8)).cuda(), K)
    torch.cuda.synchronize()
    is_reg = O.register_mask(total_rows, reg_idx)
    want, n_want = O.lambda2_for_budget(s2, ref2, keep1, is_reg, row_off, K)
    got = lam.cpu().numpy()[0]
    assert int(n.cpu()[0]) == n_want
    assert got.tobytes() == np.float32(want).tobytes(), (K, got, want)   # bit-exact: same fp32 arithmetic
    if 0 < K <= n_want:
        # the library's own threshold at lambda2* keeps at least K rows over the samples with a
        # positive reference, and fewer one fp32 step above it
        pos = torch.from_numpy(ref2 > 0).cuda()
        k1 = torch.from_numpy(keep1.astype(np.uint8)).cuda()
        r2 = torch.from_numpy(ref2).cuda()
        s2d = torch.from_numpy(s2).cuda()
        kept = []
        for lam_try in (got, np.nextafter(got, np.float32(np.inf))):
            _, cnt = occ.occam_threshold(layout, s2d, r2, occ.OCCAM_REF_SAMPLE, float(lam_try),
                                         prev_keep=k1, keep_registers=False)
            torch.cuda.synchronize()
            kept.append(int(cnt[pos].sum().item()))
        assert kept[0] >= K > kept[1], (K, kept)


@pytest.mark.parametrize("seed", [0, 1])
def test_lambda2_select_matches_oracle_random(seed):
    b = tiny_batch(B=5, segs=2, P=(300, 7, 1000, 64, 2), R=3, M=(2, 2, 2, 2, 2), seed=50 + seed)
    m = b["meta"]
    rng = np.random.default_rng(seed)
    R = m["total_rows"]
    s2 = (rng.random(R) * rng.choice([1e-4, 1e-2, 1.0], R)).astype(np.float32)
    s2[rng.random(R) < 0.05] = 0.0                          # exact zeros
    s2[10:40] = s2[10]                                      # ties
    ref2 = (rng.random(m["B"]) * 0.1).astype(np.float32)
    ref2[1] = 0.0                                           # a sample without a positive reference
    keep1 = rng.random(R) < 0.4
    n = int(keep1.sum())
    for K in (0, 1, 2, 17, n // 2, n - 1, n, n + 5, 10 ** 9):
        _lambda2_case(b, s2, ref2, keep1, K)


def test_lambda2_select_at_batch_scale():
    """192,000 rows (64 samples of 2,996 visual rows and 4 registers): every
    grid pass of the selection walks several rows per thread. Scores with
    ties, exact zeros and a few samples without a positive reference."""
    import paper_2605_29657_gb300 as occ

    B, n = 64, 3000
    row_off = np.arange(B + 1, dtype=np.int64) * n
    reg_idx = np.concatenate([b * n + n - 4 + np.arange(4) for b in range(B)]).astype(np.int32)
    layout = occ.BatchLayout(row_off, row_off.copy(), reg_idx, np.arange(B + 1) * 4, np.arange(B + 1) * 8)
    rng = np.random.default_rng(7)
    R = B * n
    s2 = (rng.random(R) * rng.choice([1e-4, 1e-2, 1.0], R)).astype(np.float32)
    s2[rng.random(R) < 0.05] = 0.0
    s2[rng.random(R) < 0.05] = np.float32(0.5)              # ties
    ref2 = (rng.random(B) * 0.01 + 1e-4).astype(np.float32)
    ref2[[3, 17]] = 0.0                                     # samples without a positive reference
    keep1 = rng.random(R) < 0.5
    n_cand = int(np.sum(keep1 & ~O.register_mask(R, reg_idx) & (ref2[np.repeat(np.arange(B), n)] > 0)))
    for K in (1, 1000, 34000, n_cand - 1, n_cand, n_cand + 1, 0):
        _lambda2_check(layout, R, reg_idx, row_off, s2, ref2, keep1, K)


def test_lambda2_select_on_oracle_scores():
    # calibration scores from the oracle (never from the CUDA path)
    b = tiny_batch(B=4, segs=2, P=(60, 13, 90, 25), R=2, M=(5, 9, 2, 30), seed=55)
    out = O.prune(b, 0.5, 1.0)
    s2 = np.asarray(out["s2"], np.float32)
    ref2 = np.asarray(out["ref2"], np.float32)
    n_vis1 = int(np.sum(out["keep1"] & ~out["is_reg"]))
    for K in (1, n_vis1 // 4, n_vis1 // 2, n_vis1):
        _lambda2_case(b, s2, ref2, out["keep1"], K)


# ----------------------------------------------------------------------------- register construction (Algorithm 1)

@pytest.mark.parametrize("case", ["tiny", "llavanext_b8"])
def test_construct_registers_matches_oracle(case):
    import paper_2605_29657_gb300 as occ

    if case == "tiny":
        b = tiny_batch(B=3, segs=2, P=(40, 7, 300), R=3, M=(5, 9, 2), hidden=96, seed=71)
        k_reg = [3, 17, 95, 40]
    else:
        b = make_batch(get_config(case), "cpu")
        k_reg = [7, 100, 511, 1000, 2047, 2048, 3000, 3333, 4000, 4095]   # 10 register channels
    m = b["meta"]
    h = b["hidden"].clone()
    rng = np.random.default_rng(3)
    for r in rng.choice(m["total_rows"], 20, replace=False):
        h[r, k_reg[0]] = 60.0                                          # sink-like activations
    want = O.construct_registers(h, m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"], np.array(k_reg))
    layout = occ.BatchLayout.from_batch(b, "cuda")
    hd = h.cuda()
    occ.occam_construct_registers(layout, hd, torch.tensor(k_reg, dtype=torch.int32, device="cuda"))
    torch.cuda.synchronize()
    got = hd.cpu().to(torch.float64).numpy()
    assert np.array_equal(got, want)                                   # exact
