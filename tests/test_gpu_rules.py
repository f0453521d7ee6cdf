"""CUDA path against the CPU oracle for the rule variants of the paper's
component ablation: the mean-threshold reference and the fixed per-sample
budget (the top-K rule of Sec. 2), as entry points of their own and as
occam_prune's rule."""

from __future__ import annotations

import numpy as np
import pytest
import torch

from oracle import occam_oracle as O
from synth import get_config, make_batch, tiny_batch
from tests.gpu_helpers import check_prune, run_prune

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


def _scores(m, seed):
    rng = np.random.default_rng(seed)
    R = m["total_rows"]
    s = (rng.random(R) * rng.choice([1e-4, 1e-2, 1.0], R)).astype(np.float32)
    s[rng.random(R) < 0.05] = 0.0                            # exact zeros
    s[10:60] = s[10]                                         # a run of ties
    prev = rng.random(R) < 0.6
    return s, prev


@pytest.mark.parametrize("seed", [0, 1])
@pytest.mark.parametrize("with_prev", [True, False])
def test_budget_keep_matches_oracle(seed, with_prev):
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=5, segs=2, P=(300, 7, 1800, 64, 2), R=3, M=(2, 2, 2, 2, 2), seed=70 + seed)
    m = b["meta"]
    s, prev = _scores(m, seed)
    if not with_prev:
        prev = np.ones_like(prev)
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    layout = occ.BatchLayout.from_batch(b, "cuda")
    ro = m["row_off_host"]
    for budget in ([0, 1, 2, 3, 4], [5, 1000, 700, -3, 1], [10 ** 6] * 5, [37, 0, 1799, 20, 0]):
        bud = np.array(budget, np.int64)
        for keep_registers in (True, False):
            keep, cnt = occ.occam_budget_keep(layout, torch.from_numpy(s).cuda(), torch.tensor(bud, dtype=torch.int32).cuda(),
                                              prev_keep=torch.from_numpy(prev.astype(np.uint8)).cuda() if with_prev else None,
                                              keep_registers=keep_registers)
            torch.cuda.synchronize()
            want, wcnt = O.budget_keep(s.astype(np.float64), ro, prev, bud, is_reg, keep_registers=keep_registers)
            assert np.array_equal(keep.cpu().numpy().astype(bool), want), (budget, keep_registers)
            assert cnt.cpu().tolist() == wcnt.tolist()


@pytest.mark.parametrize("scope", [0, 1])
@pytest.mark.parametrize("with_prev", [True, False])
def test_mean_reference_matches_oracle(scope, with_prev):
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=4, segs=3, P=(300, 7, 1800, 64), R=2, M=(2, 2, 2, 2), seed=80)
    m = b["meta"]
    s, prev = _scores(m, 3)
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    layout = occ.BatchLayout.from_batch(b, "cuda")
    off = m["seg_off_host"] if scope == occ.OCCAM_REF_SEGMENT else m["row_off_host"]
    cand = ~is_reg & (prev if with_prev else True)
    pk = torch.from_numpy(prev.astype(np.uint8)).cuda() if with_prev else None
    ref = occ.occam_mean_reference(layout, torch.from_numpy(s).cuda(), scope, prev_keep=pk)
    torch.cuda.synchronize()
    want = O.mean_reference(s.astype(np.float64), off, cand)
    # an fp64 sum rounded once to fp32
    np.testing.assert_allclose(ref.cpu().numpy(), want, rtol=2 ** -23, atol=0)


CASES = [
    ("ragged_three", dict(B=3, segs=2, P=(5, 37, 130), R=2, M=(1, 7, 70), seed=2), 0.4, 1.1),
    ("text_tiles", dict(B=2, segs=3, P=(200, 90), R=4, M=(64, 129), seed=3), 0.3, 1.3),
    ("fused_c8", dict(B=2, segs=1, P=(1000, 1532), R=4, M=(130, 33), seed=25), 0.0, 1.15),
    ("mixed_paths", dict(B=2, segs=1, P=(1700, 200), R=3, M=(70, 90), seed=23), 0.0, 1.1),
]


def _budget_for(b, frac, seed):
    """Per-sample budgets: a fraction of the sample's rows, plus a 0 and an oversize entry."""
    m = b["meta"]
    rows = np.diff(m["row_off_host"])
    bud = np.maximum(1, (rows * frac).astype(np.int64))
    if len(bud) > 1:
        bud[0] = 0
        bud[-1] = rows[-1] * 2
    return bud


@pytest.mark.parametrize("rule", ["mean", "budget"])
@pytest.mark.parametrize("name,kw,l1,l2", CASES, ids=[c[0] for c in CASES])
def test_prune_rule_matches_oracle(name, kw, l1, l2, rule):
    b = _tiny(**kw)
    budget = _budget_for(b, 0.1, 0) if rule == "budget" else None
    # the mean references are larger than the register ones here: a smaller lambda keeps a fair share
    l1m, l2m = (l1 * 0.5, l2 * 0.5) if rule == "mean" else (l1, l2)
    gpu = run_prune(b, l1m, l2m, rule=rule, budget=budget)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, l1m, l2m, rule=rule, budget=budget)
    assert rep["kept"] > 0


@pytest.mark.parametrize("rule", ["mean", "budget"])
def test_prune_rule_twopass_and_mutual(rule):
    b = _tiny(B=3, segs=1, P=(60, 301, 150), R=4, M=(5, 90, 64), stage1="mutual", d1=72, seed=6,
              query_bias=0.5, beta1=2.0)
    budget = _budget_for(b, 0.2, 1) if rule == "budget" else None
    for path in ("auto", "twopass"):
        gpu = run_prune(b, 0.5, 1.1, rule=rule, budget=budget, path=path)
        assert gpu["status"] == 0
        check_prune(b, gpu, 0.5, 1.1, rule=rule, budget=budget)


@pytest.mark.parametrize("rule", ["mean", "budget"])
@pytest.mark.parametrize("name", ["llava15_b1", "llavanext_b8"])
def test_prune_rule_small_workloads(name, rule):
    w = get_config(name)
    b = make_batch(w)
    budget = None
    if rule == "budget":
        budget = np.full(b["meta"]["B"], int(w.targets.get("count_vis", 64)), np.int64)
    gpu = run_prune(b, w.lambda1, w.lambda2, rule=rule, budget=budget)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, w.lambda1, w.lambda2, rule=rule, budget=budget)
    if rule == "budget":
        n1 = gpu["n1_vis"]
        assert gpu["count_vis"].tolist() == np.minimum(budget, n1).tolist()
    print(name, rule, rep)


# ----------------------------------------------------------------------------- grouped-query Stage II

GQA_CASES = [
    ("gqa_ragged", dict(B=3, segs=2, P=(5, 37, 130), R=2, M=(1, 7, 70), seed=31, H2kv=8), 0.4, 1.1),
    ("gqa_c8", dict(B=2, segs=1, P=(1000, 1532), R=4, M=(130, 33), seed=32, H2kv=8), 0.0, 1.15),
    ("gqa_mixed", dict(B=2, segs=1, P=(1700, 200), R=3, M=(70, 90), seed=33, H2kv=4), 0.0, 1.1),
    ("gqa_one_kv_head", dict(B=2, segs=2, P=(200, 90), R=4, M=(64, 129), seed=34, H2kv=1), 0.3, 1.3),
]


@pytest.mark.parametrize("path", ["auto", "narrow", "twopass"])
@pytest.mark.parametrize("name,kw,l1,l2", GQA_CASES, ids=[c[0] for c in GQA_CASES])
def test_prune_grouped_query_matches_oracle(name, kw, l1, l2, path):
    b = _tiny(**kw)
    assert b["K2"].shape[1] == kw["H2kv"] and b["Q_text"].shape[1] == 32
    gpu = run_prune(b, l1, l2, path=path)
    assert gpu["status"] == 0
    rep = check_prune(b, gpu, l1, l2)
    assert rep["kept"] > 0


def test_grouped_query_text_keys_none():
    b = _tiny(B=2, segs=1, P=(40, 70), R=2, M=(12, 3), seed=35, H2kv=8)
    gpu = run_prune(b, 0.3, 1.0, text_keys=False)
    check_prune(b, gpu, 0.3, 1.0, text_keys="none")


def test_grouped_query_workload_shape():
    """LLaVA-NeXT-shaped batch of 8 with 8 key heads (a grouped-query LLM layer)."""
    from dataclasses import replace
    w = replace(get_config("llavanext_b8"), H2kv=8)
    b = make_batch(w)
    gpu = run_prune(b, w.lambda1, w.lambda2)
    assert gpu["status"] == 0
    check_prune(b, gpu, w.lambda1, w.lambda2)


def test_kv_heads_must_divide_query_heads():
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=1, segs=1, P=(20,), R=2, M=(4,), seed=36)
    g = {k: v.cuda() for k, v in b.items() if isinstance(v, torch.Tensor) and v.dtype == torch.bfloat16}
    layout = occ.BatchLayout.from_batch(b, "cuda")
    keep1 = torch.ones(b["meta"]["total_rows"], dtype=torch.uint8, device="cuda")
    bad = g["K2"][:, :12].contiguous()                       # 12 key heads for 32 query heads
    with pytest.raises(occ.OccamError):
        occ.occam_score_stage2(layout, g["Q_text"], bad, keep1, K_text=g["K_text"][:, :12].contiguous())


# ----------------------------------------------------------------------------- combinations with host inputs

@pytest.mark.parametrize("variant", ["gqa", "budget", "mean"])
def test_host_inputs_with_variants(variant):
    """occam_prune_staged (K2, hidden, V in pinned host memory) under grouped-query keys and under both
    rule variants: bit-identical to the all-device call, and under the parity rule against the oracle."""
    kw = dict(B=3, segs=2, P=(120, 57, 300), R=3, M=(70, 5, 130), seed=41)
    if variant == "gqa":
        kw["H2kv"] = 8
    b = _tiny(**kw)
    rule = "register" if variant == "gqa" else variant
    budget = _budget_for(b, 0.15, 2) if variant == "budget" else None
    l1, l2 = (0.1, 0.6) if variant == "mean" else (0.2, 1.2)
    dev = run_prune(b, l1, l2, rule=rule, budget=budget)
    host = run_prune(b, l1, l2, rule=rule, budget=budget, host_inputs=True)
    assert host["status"] == 0 and dev["status"] == 0
    for k in ("s1", "ref1", "s2", "ref2", "keep1", "keep2", "count_vis", "count_out", "out_off", "n1_vis"):
        assert np.array_equal(host[k], dev[k]), k
    kept = int(dev["out_off"][-1])
    assert np.array_equal(host["out_index"][:kept], dev["out_index"][:kept])
    for a, c in zip(host["gathered"], dev["gathered"]):
        assert torch.equal(a[:kept], c[:kept])
    check_prune(b, host, l1, l2, rule=rule, budget=budget)


def test_rules_capture_into_a_graph_and_replay_identically():
    """occam_prune under each rule inside a CUDA graph: a replay reproduces the eager outputs."""
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=3, segs=2, P=(100, 57, 220), R=3, M=(70, 5, 130), seed=42)
    g = {k: v.cuda() for k, v in b.items() if isinstance(v, torch.Tensor) and v.dtype == torch.bfloat16}
    layout = occ.BatchLayout.from_batch(b, "cuda")
    st1 = dict(mode="cls", q=g["q_cls"], k_cls=g["k_cls"], K1=g["K1"])
    st2 = dict(Q_text=g["Q_text"], K_text=g["K_text"], K2=g["K2"])
    budget = torch.tensor(_budget_for(b, 0.1, 3), dtype=torch.int32, device="cuda")
    for rule in ("register", "mean", "budget"):
        call = occ.PruneCall(layout, st1, st2, 0.2, 1.2, gather=(g["hidden"],), rule=rule,
                             budget=budget if rule == "budget" else None)
        call()
        torch.cuda.synchronize()
        want = {k: v.clone() for k, v in call.out.items()}
        cs = torch.cuda.Stream()
        cs.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cs):
            call(cs)
        torch.cuda.current_stream().wait_stream(cs)
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            call()
        for k in call.out:
            call.out[k].zero_()
        graph.replay()
        torch.cuda.synchronize()
        assert call.status() == 0
        kept = int(want["out_off"][-1])
        for k, v in want.items():
            if k == "out_index":
                assert torch.equal(v[:kept], call.out[k][:kept]), (rule, k)
            else:
                assert torch.equal(v, call.out[k]), (rule, k)


# ----------------------------------------------------------------------------- merged-token pooling

@pytest.mark.parametrize("mode", ["sum", "mean", "max"])
@pytest.mark.parametrize("group", [1, 4, 16])
def test_pool_scores_matches_oracle(mode, group):
    import paper_2605_29657_gb300 as occ

    rng = np.random.default_rng(group)
    s = (rng.random(4 * 16 * 777) * rng.choice([1e-5, 1e-2, 1.0], 4 * 16 * 777)).astype(np.float32)
    got = occ.occam_pool_scores(torch.from_numpy(s).cuda(), group, mode).cpu().numpy()
    want = O.pool_scores(s.astype(np.float64), group, mode)
    if mode == "max":
        assert np.array_equal(got.astype(np.float64), want)
    else:
        # fp32 additions of `group` values in row order
        np.testing.assert_allclose(got, want, rtol=group * 2 ** -23, atol=0)


def test_pool_scores_of_mutual_stage1():
    """Stage-I mutual scores of patch rows pooled 4 to 1 (a 2x2 merger) match the oracle's pooled scores."""
    import paper_2605_29657_gb300 as occ

    b = _tiny(B=2, segs=1, P=(60, 124), R=4, M=(3, 3), stage1="mutual", d1=72, seed=43, query_bias=0.5)
    m = b["meta"]
    layout = occ.BatchLayout.from_batch(b, "cuda")
    s1, _ = occ.occam_score_stage1(layout, occ.OCCAM_STAGE1_MUTUAL, b["Q1"].cuda(), b["K1"].cuda())
    pooled = occ.occam_pool_scores(s1, 4, "sum").cpu().numpy()
    ref1, _ = O.stage1_mutual(b["Q1"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    np.testing.assert_allclose(pooled, O.pool_scores(ref1, 4, "sum"), rtol=1e-3, atol=1e-5)


def test_pool_scores_rejects_ragged_groups():
    import paper_2605_29657_gb300 as occ

    with pytest.raises(occ.OccamError):
        occ.occam_pool_scores(torch.zeros(10, device="cuda"), 4)
