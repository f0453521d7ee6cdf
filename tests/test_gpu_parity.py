"""CUDA path (through the C ABI) against the CPU oracle on seeded inputs.

Sizes are small enough for the oracle to finish in seconds but span several
tiles of every kernel (Stage-II text tiles of 64 rows and key chunks of 128,
[CLS] cluster shares, 2,048-row scan tiles) with ragged tails.
"""

from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import occam_oracle as O
from synth import get_config, make_batch, tiny_batch
from tests.gpu_helpers import check_prune, close, run_prune, to_device

pytestmark = pytest.mark.gpu

H = dict(H1=16, d1=64, H2=32, d2=128)


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _tiny(**kw):
    args = dict(H, hidden=256, beta1=2.0, sinks=("count", 1))
    args.update(kw)
    return tiny_batch(**args)


CASES = [
    # (name, tiny_batch kwargs, lambda1, lambda2)
    ("one_segment_small", dict(B=1, segs=1, P=(9,), R=1, M=(3,), seed=1), 0.5, 1.0),
    ("ragged_three", dict(B=3, segs=2, P=(5, 37, 130), R=2, M=(1, 7, 70), seed=2), 0.4, 1.1),
    ("text_tiles", dict(B=2, segs=3, P=(200, 90), R=4, M=(64, 129), seed=3), 0.3, 1.3),
    ("key_chunks", dict(B=2, segs=1, P=(700, 300), R=3, M=(20, 5), seed=4), 0.05, 1.2),
    ("scan_tiles", dict(B=5, segs=2, P=(500, 333, 612, 47, 401), R=4, M=(9, 33, 65, 2, 17), seed=5), 0.2, 1.05),
    # fused tensor-core Stage II: text tiles of 128 rows, chunk edges at 64 keys per CTA
    ("fused_text_edges", dict(B=4, segs=1, P=(252, 60, 300, 5), R=4, M=(128, 129, 256, 1), seed=21), 0.0, 1.1),
    ("fused_max_keys", dict(B=1, segs=1, P=(764,), R=4, M=(40,), seed=22), 0.0, 1.2),
    # 8-CTA clusters: S1 above 768 keys, up to their limit of 1536
    ("fused_c8", dict(B=2, segs=1, P=(1000, 1532), R=4, M=(130, 33), seed=25), 0.0, 1.15),
    # one sample above the fused kernel's S1 limit (two-pass), one below (fused)
    ("mixed_paths", dict(B=2, segs=1, P=(1700, 200), R=3, M=(70, 90), seed=23), 0.0, 1.1),
    # many key ranges (the two-pass statistics pass caps them at 16) over
    # 128-row statistics tiles with ragged last tiles (M = 200, 257)
    ("twopass_ranges", dict(B=2, segs=1, P=(1300, 2900), R=4, M=(200, 257), seed=26), 0.0, 1.1),
]


@pytest.mark.parametrize("path", ["auto", "narrow", "twopass"])
@pytest.mark.parametrize("name,kw,l1,l2", CASES, ids=[c[0] for c in CASES])
def test_prune_cls_matches_oracle(name, kw, l1, l2, path):
    b = _tiny(**kw)
    gpu = run_prune(b, l1, l2, path=path)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, l1, l2)
    assert rep["kept"] > 0


def test_registers_only_s1():
    """Stage I keeps no visual row: S1 = registers (some CTAs of a cluster own no keys)."""
    b = _tiny(B=2, segs=1, P=(30, 9), R=1, M=(5, 140), seed=24)
    gpu = run_prune(b, 1e9, 1.0)
    assert gpu["status"] == 0
    check_prune(b, gpu, 1e9, 1.0)


@pytest.mark.parametrize("d1", [72, 64])
def test_prune_mutual_matches_oracle(d1):
    b = _tiny(B=3, segs=1, P=(60, 301, 150), R=4, M=(5, 90, 64), stage1="mutual", d1=d1, seed=6,
              query_bias=0.5, beta1=2.0)
    gpu = run_prune(b, 0.5, 1.1)
    assert gpu["status"] == 0
    check_prune(b, gpu, 0.5, 1.1)


@pytest.mark.parametrize("d1", [72, 128])
def test_prune_cls_head_dims(d1):
    """[CLS] mode with vision heads of 72 and 128 dims (2,304- and 4,096-byte
    K1 rows; 72 takes 18-byte lane slices), ragged segments and tiles."""
    b = _tiny(B=3, segs=2, P=(200, 37, 130), R=3, M=(9, 70, 129), d1=d1, seed=35)
    for path in ("auto", "twopass"):
        gpu = run_prune(b, 0.3, 1.2, path=path)
        assert gpu["status"] == 0
        rep = check_prune(b, gpu, 0.3, 1.2)
        assert rep["kept"] > 0


@pytest.mark.parametrize("d1", [72, 64, 80])
def test_prune_mutual_segment_edges(d1):
    """Mutual Stage I on segments of 5 rows (one partial key block), 133 (a
    second 128-row tile of one row past the first), 260 (a second 256-key
    block) and 512 (whole tiles and blocks), for each supported d1 (72 takes
    the log-sums folded into the MMA, 64 and 80 the shared-memory ring)."""
    b = _tiny(B=4, segs=1, P=(1, 129, 256, 508), R=4, M=(3, 40, 17, 128), stage1="mutual", d1=d1, seed=33,
              query_bias=0.5, beta1=2.0)
    gpu = run_prune(b, 0.5, 1.1)
    assert gpu["status"] == 0
    check_prune(b, gpu, 0.5, 1.1)


@pytest.mark.parametrize("d1", [72, 64])
def test_prune_mutual_late_large_logits(d1):
    """Keys past the first 256 of a segment with logits far above the first
    block's (their K1 rows scaled by 64, exactly in bf16; about 340 in log2
    units above it): the first mutual pass's online softmax rescales its
    running sums by 2^-340 and below, and the scores still match the oracle."""
    b = _tiny(B=2, segs=1, P=(700, 300), R=4, M=(20, 50), stage1="mutual", d1=d1, seed=31, query_bias=0.5,
              beta1=2.0)
    m = b["meta"]
    a, z = int(m["seg_off_host"][0]), int(m["seg_off_host"][1])
    K1 = b["K1"]
    K1[a + 256:z] = (K1[a + 256:z].float() * 64).to(K1.dtype)
    gpu = run_prune(b, 0.5, 1.1)
    assert gpu["status"] == 0
    check_prune(b, gpu, 0.5, 1.1)


@pytest.mark.parametrize("lam1", [0.3, 0.0])
def test_segment_above_finalize_staging(lam1):
    """A [CLS] segment of 23,004 rows, above the 22,400 whose s1 and roles the
    finalize kernel stages in shared memory (it works from global memory),
    with a small sample beside it; at lambda1 = 0 every row enters S1 and
    Stage II takes the two-pass path for the large sample."""
    b = _tiny(B=2, segs=1, P=(23000, 40), R=4, M=(8, 5), hidden=32, seed=51)
    gpu = run_prune(b, lam1, 1.1)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, lam1, 1.1)
    assert rep["kept"] > 0


@pytest.mark.parametrize("B", [300, 2100])
def test_many_samples(B):
    """More samples than the planning CTA's 256 threads (the plan walks them
    in chunks) and, at 2,100, more than the 2,048 whose row offsets and
    thresholds the scan stages in shared memory; samples of 0-11 visual rows
    and one register."""
    rng = np.random.default_rng(B)
    P = tuple(int(x) for x in rng.integers(0, 12, size=B))
    M = tuple(int(x) for x in rng.integers(1, 20, size=B))
    b = _tiny(B=B, segs=1, P=P, R=1, M=M, hidden=32, seed=50, sinks=("count", 0))
    gpu = run_prune(b, 0.3, 1.1)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, 0.3, 1.1)
    assert rep["kept"] > 0


@pytest.mark.parametrize("name", ["llava15_b1", "llavanext_b8"])
def test_small_workloads(name):
    w = get_config(name)
    b = make_batch(w)
    gpu = run_prune(b, w.lambda1, w.lambda2)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, w.lambda1, w.lambda2)
    print(name, rep)


# ----------------------------------------------------------------------------- edge cases

def test_lambda_zero_keeps_everything_and_copies_bits():
    b = _tiny(B=2, segs=2, P=(30, 11), R=2, M=(4, 9), seed=7)
    gpu = run_prune(b, 0.0, 0.0)
    check_prune(b, gpu, 0.0, 0.0)
    n = b["meta"]["total_rows"]
    assert gpu["out_index"][:n].tolist() == list(range(n))
    for t, name in zip(gpu["gathered"], ("hidden", "K2", "V")):
        src = b[name].reshape(n, -1)
        assert torch.equal(t[:n].view(torch.int16), src.view(torch.int16))


def test_empty_stage1_keeps_only_registers():
    b = _tiny(B=2, segs=2, P=(20, 13), R=3, M=(5, 6), seed=8)
    gpu = run_prune(b, 1e9, 1.0)
    check_prune(b, gpu, 1e9, 1.0)
    assert gpu["count_vis"].tolist() == [0, 0]
    assert gpu["n1_vis"].tolist() == [0, 0]
    assert gpu["count_out"].tolist() == [6, 6]


@pytest.mark.parametrize("keep_registers", [False, True])
def test_keep_registers_flag(keep_registers):
    b = _tiny(B=2, segs=2, P=(25, 40), R=2, M=(8, 3), seed=9)
    gpu = run_prune(b, 0.3, 1.0, keep_registers=keep_registers)
    check_prune(b, gpu, 0.3, 1.0, keep_registers=keep_registers)


def test_capacity_overflow_reports_and_stays_in_bounds():
    b = _tiny(B=2, segs=1, P=(50, 60), R=2, M=(4, 4), seed=10)
    cap = 7
    gpu = run_prune(b, 0.0, 0.0, capacity_rows=cap)
    assert gpu["status"] == 2  # OCCAM_ERR_CAPACITY
    check_prune(b, gpu, 0.0, 0.0, capacity_rows=cap)
    assert int(gpu["out_off"][-1]) == b["meta"]["total_rows"]


@pytest.mark.parametrize("path", ["auto", "twopass"])
def test_text_keys_none(path):
    b = _tiny(B=2, segs=1, P=(40, 70), R=2, M=(12, 3), seed=11)
    gpu = run_prune(b, 0.3, 1.0, text_keys=False, path=path)
    check_prune(b, gpu, 0.3, 1.0, text_keys="none")


def test_deterministic_across_calls():
    b = _tiny(B=3, segs=2, P=(100, 57, 220), R=3, M=(70, 5, 130), seed=12)
    a = run_prune(b, 0.2, 1.2)
    c = run_prune(b, 0.2, 1.2)
    for k in ("s1", "ref1", "s2", "ref2", "keep1", "keep2", "out_index", "count_out", "out_off"):
        assert np.array_equal(a[k], c[k]), k


@pytest.mark.parametrize("path", ["auto", "twopass"])
def test_host_inputs_match_device_inputs(path):
    # K2, hidden and V in pinned host memory (occam_prune_staged): only S1
    # rows of K2 and the kept rows are read across the host link, and every
    # output is bit-identical to the all-device call
    b = _tiny(B=4, segs=2, P=(120, 57, 300, 9), R=3, M=(70, 5, 130, 1), seed=21)
    dev = run_prune(b, 0.2, 1.2, path=path)
    host = run_prune(b, 0.2, 1.2, path=path, host_inputs=True)
    assert host["status"] == 0
    for k in ("s1", "ref1", "s2", "ref2", "keep1", "keep2", "count_vis", "count_out", "out_off", "n1_vis"):
        assert np.array_equal(host[k], dev[k]), k
    kept = int(dev["out_off"][-1])
    assert np.array_equal(host["out_index"][:kept], dev["out_index"][:kept])
    for a, c in zip(host["gathered"], dev["gathered"]):
        assert torch.equal(a[:kept], c[:kept])
    check_prune(b, host, 0.2, 1.2)


def test_host_inputs_refuse_pageable_memory():
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=2, segs=1, P=(30, 40), R=2, M=(4, 6), seed=22)
    g = to_device(b, "cuda")
    layout = occ.BatchLayout.from_batch(b, "cuda")
    st1 = dict(mode="cls", q=g["q_cls"], k_cls=g["k_cls"], K1=g["K1"])
    # pageable host K2: refused by the binding before any launch
    with pytest.raises(occ.OccamError):
        occ.occam_prune(layout, st1, dict(Q_text=g["Q_text"], K_text=g["K_text"], K2=g["K2"].cpu()), 0.2, 1.0,
                        host_inputs=True)
    # ... and by the library itself when handed one through the C ABI
    call = occ.PruneCall(layout, st1, dict(Q_text=g["Q_text"], K_text=g["K_text"], K2=g["K2"].cpu().pin_memory()),
                         0.2, 1.0, host_inputs=True)
    pageable = g["K2"].cpu()
    call.args.stage2.K2 = pageable.data_ptr()
    with pytest.raises(occ.OccamError) as e:
        call()
    assert e.value.code == occ._lib.OCCAM_ERR_INVALID_ARG
    # a host tensor where the library requires device memory (a TMA-read input)
    call2 = occ.PruneCall(layout, st1, dict(Q_text=g["Q_text"], K_text=g["K_text"], K2=g["K2"]), 0.2, 1.0)
    pinned = g["K2"].cpu().pin_memory()
    call2.args.stage2.K2 = pinned.data_ptr()
    with pytest.raises(occ.OccamError) as e:
        call2()
    assert e.value.code == occ._lib.OCCAM_ERR_INVALID_ARG


# ----------------------------------------------------------------------------- standalone entry points

def test_standalone_entry_points():
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=3, segs=2, P=(33, 80, 7), R=2, M=(6, 70, 2), seed=13)
    m = b["meta"]
    dev = torch.device("cuda")
    layout = occ.BatchLayout.from_batch(b, dev)
    g = {k: b[k].to(dev) for k in ("q_cls", "k_cls", "K1", "Q_text", "K_text", "K2", "hidden")}
    s1, ref1 = occ.occam_score_stage1(layout, occ.OCCAM_STAGE1_CLS, g["q_cls"], g["K1"], k_cls=g["k_cls"])
    os1, oref1 = O.stage1_cls(b["q_cls"], b["k_cls"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    close("s1", s1.cpu().numpy(), os1)
    close("ref1", ref1.cpu().numpy(), oref1)
    # threshold on the oracle's own scores (fp32 copies): exact outside the band
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    seg_of_row = np.repeat(np.arange(m["S_tot"]), np.diff(m["seg_off_host"]))
    s_t = torch.tensor(os1, dtype=torch.float32, device=dev)
    r_t = torch.tensor(oref1, dtype=torch.float32, device=dev)
    keep, cnt = occ.occam_threshold(layout, s_t, r_t, occ.OCCAM_REF_SEGMENT, 0.6, keep_registers=True)
    s32 = s_t.cpu().numpy().astype(np.float64)
    tau32 = (np.float32(0.6) * r_t.cpu().numpy())[seg_of_row].astype(np.float64)
    want = ((s32 >= tau32) & ~is_reg) | is_reg
    assert np.array_equal(keep.cpu().numpy().astype(bool), want)
    assert cnt.cpu().tolist() == [int((want & ~is_reg)[a:z].sum()) for a, z in zip(m["row_off_host"][:-1], m["row_off_host"][1:])]
    # Stage II on a given S1 mask
    rng = np.random.default_rng(0)
    keep1 = (rng.random(m["total_rows"]) < 0.5) | is_reg
    k1 = torch.tensor(keep1.astype(np.uint8), device=dev)
    s2, ref2 = occ.occam_score_stage2(layout, g["Q_text"], g["K2"], k1, K_text=g["K_text"])
    os2, oref2 = O.stage2_scores(b["Q_text"], b["K_text"], b["K2"], keep1, is_reg, m["row_off_host"], m["text_off_host"])
    close("s2", s2.cpu().numpy(), os2)
    close("ref2", ref2.cpu().numpy(), oref2)
    # compaction of a random mask with one gather tensor
    mask = rng.random(m["total_rows"]) < 0.3
    mk = torch.tensor(mask.astype(np.uint8), device=dev)
    res = occ.occam_compact(layout, mk, tensors=(g["hidden"],))
    oi, oc, oo, og = O.compact(mask, m["row_off_host"], [b["hidden"].view(torch.int16).numpy()])
    n = int(oo[-1])
    assert res["out_index"][:n].cpu().tolist() == oi.tolist()
    assert res["count_out"].cpu().tolist() == oc.tolist()
    assert res["out_off"].cpu().tolist() == oo.tolist()
    assert np.array_equal(res["gathered"][0][:n].cpu().view(torch.int16).numpy(), og[0])


def test_invalid_arguments_raise():
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=1, segs=1, P=(10,), R=1, M=(2,), seed=14)
    dev = torch.device("cuda")
    layout = occ.BatchLayout.from_batch(b, dev)
    g = {k: b[k].to(dev) for k in ("q_cls", "K1")}
    with pytest.raises(occ.OccamError):
        occ.occam_score_stage1(layout, occ.OCCAM_STAGE1_CLS, g["q_cls"], g["K1"][:, :8].contiguous())
    with pytest.raises(occ.OccamError):
        occ.occam_score_stage1(layout, occ.OCCAM_STAGE1_CLS, g["q_cls"].float(), g["K1"])


# ----------------------------------------------------------------------------- shapes beyond the workloads

@pytest.mark.parametrize("H2", [2, 8, 64])
def test_other_llm_head_counts(H2):
    """H2 = 2 takes the two-pass path (the fused kernel needs at least 4 heads); 8 and 64 the fused one."""
    b = tiny_batch(B=2, segs=2, P=(90, 41), R=2, M=(70, 9), H1=16, d1=64, H2=H2, d2=128, hidden=64, seed=61,
                   beta1=2.0)
    for path in ("auto", "twopass"):
        gpu = run_prune(b, 0.3, 1.1, path=path)
        assert gpu["status"] == 0
        check_prune(b, gpu, 0.3, 1.1)


def test_many_small_samples():
    """More samples than one planning block holds (257 > 256 threads), one-token texts, tiny segments."""
    B = 257
    rng = np.random.default_rng(62)
    P = tuple(int(x) for x in rng.integers(1, 12, B))
    M = tuple(int(x) for x in rng.integers(1, 4, B))
    b = tiny_batch(B=B, segs=1, P=P, R=1, M=M, H1=16, d1=64, H2=32, d2=128, hidden=32, seed=62, beta1=2.0)
    gpu = run_prune(b, 0.4, 1.0)
    assert gpu["status"] == 0
    check_prune(b, gpu, 0.4, 1.0)


def test_long_text_many_fused_items():
    """Text of 600 tokens: five 128-row fused items (and ten 64-row two-pass tiles) for one sample."""
    b = _tiny(B=2, segs=1, P=(300, 40), R=4, M=(600, 3), seed=63)
    for path in ("auto", "narrow", "twopass"):
        gpu = run_prune(b, 0.2, 1.2, path=path)
        assert gpu["status"] == 0
        check_prune(b, gpu, 0.2, 1.2)


@pytest.mark.parametrize("name", ["llava15_b1", "llavanext_b8", "llavanext_b64"])
def test_kernel_count_matches_profiler(name):
    """occam_last_call_kernels agrees with the kernels a profiler sees for one prune call."""
    import paper_2605_29657_gb300 as occ
    from torch.profiler import ProfilerActivity, profile

    w = get_config(name)
    b = make_batch(w, "cuda", with_gather=True)
    layout = occ.BatchLayout.from_batch(b, "cuda")
    call = occ.PruneCall(layout, dict(mode="cls", q=b["q_cls"], k_cls=b["k_cls"], K1=b["K1"]),
                         dict(Q_text=b["Q_text"], K_text=b["K_text"], K2=b["K2"]), w.lambda1, w.lambda2,
                         gather=(b["hidden"],))
    call()
    torch.cuda.synchronize()
    for _ in range(2):  # a process's first profiling session may miss device activity
        with profile(activities=[ProfilerActivity.CUDA]) as prof:
            call()
            torch.cuda.synchronize()
    claimed = occ.occam_last_call_kernels()
    ours = [e for e in prof.events() if e.device_type == torch.autograd.DeviceType.CUDA and "occam" in e.name]
    if not ours:
        pytest.skip("the profiler sees no device activity here")
    assert len(ours) == claimed, (claimed, sorted(e.name for e in ours))
    assert call.status() == 0
