"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each pin is chosen so that a plausible mistake in the oracle fails it:
a dropped [CLS] key, '>' instead of '>=', a non-causal or wrong Stage-II key
set, mean instead of max over text tokens, a register counted as a
candidate, a per-sample instead of per-segment Stage-I threshold, a wrong
head average, a reordered or lossy gather.
"""

from __future__ import annotations

import math
from decimal import Decimal, getcontext

import numpy as np
import pytest
import torch

from oracle import occam_oracle as O
from synth import tiny_batch
from tests._fixtures import worked_example


# ----------------------------------------------------------------------------- worked example

@pytest.mark.parametrize("case", [0, 1, 2])
def test_worked_example_hand_derived(case):
    """Hand-derived example (tests/golden/worked_example.json; Eqs. 4-8)."""
    batch, g = worked_example()
    c = g["cases"][case]
    out = O.prune(batch, g["lambda1"], c["lambda2"])
    e = math.e
    Z1 = 3 + e + e * e
    np.testing.assert_allclose(out["s1"], [e / Z1, 1 / Z1, e * e / Z1, 1 / Z1], rtol=1e-14)
    np.testing.assert_allclose(out["ref1"], [1 / Z1], rtol=1e-14)
    assert out["keep1"].astype(int).tolist() == c["keep1"]
    s2_r0 = e / (e + 3)
    s2_r2 = e * e / (3 + e + e * e)
    ref2 = (1 / (e + 3) + 1 / (3 + e + e * e)) / 2
    np.testing.assert_allclose(out["s2"][[0, 2]], [s2_r0, s2_r2], rtol=1e-14)
    assert out["s2"][1] == 0.0  # pruned in Stage I: never scored in Stage II
    np.testing.assert_allclose(out["ref2"], [ref2], rtol=1e-14)
    assert out["keep2"].astype(int).tolist() == c["keep2"]
    assert int(out["count_vis"][0]) == c["count_vis"]
    assert out["out_index"].tolist() == c["out_index"]
    assert out["count_out"].tolist() == [len(c["out_index"])]


# ----------------------------------------------------------------------------- P1 softmax

def test_softmax_rows_sum_to_one():
    rng = np.random.default_rng(0)
    x = rng.normal(size=(50, 77)) * 20
    A = O.softmax(x, axis=1)
    np.testing.assert_allclose(A.sum(axis=1), 1.0, atol=1e-12)
    assert (A >= 0).all()
    # shift invariance and the textbook formula on a small row
    row = np.array([0.5, -1.0, 2.0])
    ref = np.exp(row) / np.exp(row).sum()
    np.testing.assert_allclose(O.softmax(row), ref, rtol=1e-15)
    np.testing.assert_allclose(O.softmax(row + 1000.0), ref, rtol=1e-12)


def test_stage1_mass_conservation():
    """Without k_cls every segment's s1 sums to 1; with it, to 1 - A(cls)."""
    b = tiny_batch(B=2, segs=3, P=(6, 9), R=2, M=(3, 2), seed=3)
    m = b["meta"]
    s1, _ = O.stage1_cls(b["q_cls"], None, b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    for s in range(m["S_tot"]):
        a, z = m["seg_off_host"][s], m["seg_off_host"][s + 1]
        assert abs(s1[a:z].sum() - 1.0) < 1e-12
    s1c, _ = O.stage1_cls(b["q_cls"], b["k_cls"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    for s in range(m["S_tot"]):
        a, z = m["seg_off_host"][s], m["seg_off_host"][s + 1]
        assert s1c[a:z].sum() < 1.0 - 1e-6
    # mutual: the average over queries of row-stochastic rows sums to 1
    bm = tiny_batch(B=2, segs=1, P=(7, 4), R=2, M=(2, 2), stage1="mutual", seed=4)
    mm = bm["meta"]
    s1m, _ = O.stage1_mutual(bm["Q1"], bm["K1"], mm["seg_off_host"], mm["reg_idx_host"], mm["reg_off_host"])
    for s in range(mm["S_tot"]):
        a, z = mm["seg_off_host"][s], mm["seg_off_host"][s + 1]
        assert abs(s1m[a:z].sum() - 1.0) < 1e-12


def test_stage2_mass_without_text_keys_and_one_token():
    """text_keys='none', M=1: sum_vis s2 + R * ref2 = 1 over the S1 rows."""
    b = tiny_batch(B=2, segs=2, P=(5, 6), R=2, M=(1, 1), seed=5)
    m = b["meta"]
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    keep1 = np.ones(m["total_rows"], bool)
    s2, ref2 = O.stage2_scores(b["Q_text"], b["K_text"], b["K2"], keep1, is_reg,
                               m["row_off_host"], m["text_off_host"], text_keys="none")
    for bb in range(m["B"]):
        a, z = m["row_off_host"][bb], m["row_off_host"][bb + 1]
        R_b = int(is_reg[a:z].sum())
        assert abs(s2[a:z][~is_reg[a:z]].sum() + R_b * ref2[bb] - 1.0) < 1e-12


# ----------------------------------------------------------------------------- P2 / P12 uniform

def _zero(t):
    return torch.zeros_like(t)


def test_stage1_cls_zero_query_is_uniform_and_ties_keep():
    b = tiny_batch(B=2, segs=2, P=(5, 8), R=3, M=(2, 3), seed=6)
    b["q_cls"] = _zero(b["q_cls"])
    m = b["meta"]
    s1, ref1 = O.stage1_cls(b["q_cls"], b["k_cls"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    for s in range(m["S_tot"]):
        a, z = m["seg_off_host"][s], m["seg_off_host"][s + 1]
        np.testing.assert_allclose(s1[a:z], 1.0 / (z - a + 1), rtol=1e-15)  # +1: the [CLS] key
    out_eq = O.prune(b, 1.0, 0.0)
    out_gt = O.prune(b, 1.0 + 2.0 ** -20, 0.0)
    is_reg = out_eq["is_reg"]
    assert out_eq["keep1"][~is_reg].all()          # equality keeps (>=)
    assert not out_gt["keep1"][~is_reg].any()
    assert out_gt["keep1"][is_reg].all()           # the register always stays in S1


def test_stage1_mutual_zero_query_is_uniform():
    b = tiny_batch(B=2, segs=1, P=(6, 9), R=2, M=(2, 2), stage1="mutual", seed=7)
    b["Q1"] = _zero(b["Q1"])
    m = b["meta"]
    s1, ref1 = O.stage1_mutual(b["Q1"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    for s in range(m["S_tot"]):
        a, z = m["seg_off_host"][s], m["seg_off_host"][s + 1]
        np.testing.assert_allclose(s1[a:z], 1.0 / (z - a), rtol=1e-14)
    out = O.prune(b, 1.0, 0.0)
    assert out["keep1"].all()
    out = O.prune(b, 1.0 + 1e-9, 0.0)
    assert not out["keep1"][~out["is_reg"]].any()


# ----------------------------------------------------------------------------- P3 Stage II closed form

def _harmonic(n):
    return sum(1.0 / k for k in range(1, n + 1))


@pytest.mark.parametrize("M", [1, 3, 7])
def test_stage2_zero_query_closed_form(M):
    """Q_text = 0: A_j is uniform over n image keys + (j+1) causal text keys.

    s2(v) = 1/(n+1) (its max, at j = 0); s2(r) = (H_{n+M} - H_n) / M.
    """
    b = tiny_batch(B=2, segs=2, P=(4, 6), R=2, M=(M, M), seed=8)
    b["Q_text"] = _zero(b["Q_text"])
    m = b["meta"]
    is_reg = O.register_mask(m["total_rows"], m["reg_idx_host"])
    rng = np.random.default_rng(1)
    keep1 = rng.random(m["total_rows"]) < 0.6
    s2, ref2 = O.stage2_scores(b["Q_text"], b["K_text"], b["K2"], keep1, is_reg,
                               m["row_off_host"], m["text_off_host"])
    for bb in range(m["B"]):
        a, z = m["row_off_host"][bb], m["row_off_host"][bb + 1]
        sel = (keep1[a:z] & ~is_reg[a:z])
        n = int(sel.sum() + is_reg[a:z].sum())
        np.testing.assert_allclose(s2[a:z][sel], 1.0 / (n + 1), rtol=1e-14)
        assert (s2[a:z][~sel & ~is_reg[a:z]] == 0).all()
        np.testing.assert_allclose(ref2[bb], (_harmonic(n + M) - _harmonic(n)) / M, rtol=1e-13)


# ----------------------------------------------------------------------------- P4 heads

def test_identical_heads_equal_single_head():
    b1 = tiny_batch(B=1, segs=2, P=(6,), R=2, M=(4,), H1=1, H2=1, seed=9)
    bH = dict(b1)
    for k in ("q_cls", "k_cls", "K1", "Q_text", "K_text", "K2"):
        bH[k] = b1[k].repeat(1, 3, 1)
    o1 = O.prune(b1, 0.7, 1.1)
    oH = O.prune(bH, 0.7, 1.1)
    for k in ("s1", "ref1", "s2", "ref2"):
        np.testing.assert_allclose(oH[k], o1[k], rtol=1e-13)
    assert (oH["keep2"] == o1["keep2"]).all()


# ----------------------------------------------------------------------------- P5 two keys

@pytest.mark.parametrize("dl", [-2, 0, 1, 3])
def test_two_key_threshold(dl):
    """One visual key, one register, integer logits: keep iff lambda <= exp(l_v - l_r)."""
    q = torch.tensor([[[2.0, 0, 0, 0]]]).to(torch.bfloat16)          # scale 1/2 -> logit = k[0]
    K1 = torch.tensor([[[float(dl), 1, 2, 3]], [[0.0, -1, 5, 2]]]).to(torch.bfloat16)
    seg_off = np.array([0, 2])
    s1, ref1 = O.stage1_cls(q, None, K1, seg_off, np.array([1]), np.array([0, 1]))
    ratio = math.exp(dl)
    assert abs(s1[0] / ref1[0] - ratio) < 1e-12 * ratio
    is_reg = np.array([False, True])
    for lam, want in ((ratio * (1 - 1e-9), True), (ratio * (1 + 1e-9), False)):
        keep = O.threshold(s1, np.full(2, ref1[0]), lam, is_reg)
        assert bool(keep[0]) == want and bool(keep[1])


# ----------------------------------------------------------------------------- P6 threshold set

def test_kept_set_is_top_count_per_segment_and_sample():
    b = tiny_batch(B=3, segs=3, P=(20, 13, 31), R=2, M=(5, 9, 2), seed=10)
    out = O.prune(b, 0.9, 1.2)
    m = b["meta"]
    is_reg = out["is_reg"]
    for s in range(m["S_tot"]):
        a, z = m["seg_off_host"][s], m["seg_off_host"][s + 1]
        vis = np.arange(a, z)[~is_reg[a:z]]
        k = int(out["keep1"][vis].sum())
        top = set(vis[np.argsort(-out["s1"][vis], kind="stable")[:k]].tolist())
        assert top == set(vis[out["keep1"][vis]].tolist())
    for bb in range(m["B"]):
        a, z = m["row_off_host"][bb], m["row_off_host"][bb + 1]
        cand = np.arange(a, z)[out["keep1"][a:z] & ~is_reg[a:z]]
        k = int(out["keep2"][cand].sum())
        top = set(cand[np.argsort(-out["s2"][cand], kind="stable")[:k]].tolist())
        assert top == set(cand[out["keep2"][cand]].tolist())


# ----------------------------------------------------------------------------- P7 monotone

def test_counts_monotone_in_lambda():
    b = tiny_batch(B=2, segs=2, P=(25, 18), R=2, M=(6, 4), seed=11)
    c1 = [O.prune(b, l1, 0.0)["n1_vis"].sum() for l1 in np.linspace(0, 2.5, 11)]
    assert all(x >= y for x, y in zip(c1, c1[1:]))
    assert c1[0] == 25 * 2 + 18 * 2
    base = O.prune(b, 0.8, 0.0)
    c2 = [O.prune(b, 0.8, l2, keep1_override=base["keep1"])["count_vis"].sum()
          for l2 in np.linspace(0, 4, 13)]
    assert all(x >= y for x, y in zip(c2, c2[1:]))
    assert c2[0] == base["n1_vis"].sum()


# ----------------------------------------------------------------------------- P8-P10 compaction

def test_lambda_zero_copies_everything():
    b = tiny_batch(B=2, segs=2, P=(5, 7), R=2, M=(3, 4), seed=12)
    out = O.prune(b, 0.0, 0.0)
    n = b["meta"]["total_rows"]
    assert out["out_index"].tolist() == list(range(n))
    for name in ("hidden", "K2", "V"):
        raw = b[name].reshape(n, -1).view(torch.int16).numpy()
        assert (out["gathered"][name] == raw).all()


def test_gather_equals_boolean_mask_indexing():
    b = tiny_batch(B=3, segs=2, P=(9, 4, 12), R=2, M=(3, 6, 2), seed=13)
    out = O.prune(b, 0.8, 1.1)
    m = b["meta"]
    keep = out["keep2"]
    hid = b["hidden"].float().numpy()
    got = b["hidden"].view(torch.int16).numpy()[out["out_index"]]
    pos = 0
    for bb in range(m["B"]):
        a, z = m["row_off_host"][bb], m["row_off_host"][bb + 1]
        want = hid[a:z][keep[a:z]]                       # numpy boolean-mask indexing
        n = want.shape[0]
        assert out["count_out"][bb] == n and out["out_off"][bb] == pos
        np.testing.assert_array_equal(
            torch.from_numpy(got[pos:pos + n]).view(torch.bfloat16).float().numpy(), want)
        assert (np.diff(out["out_index"][pos:pos + n]) > 0).all()   # order preserved
        pos += n
    assert out["out_off"][-1] == pos == keep.sum()


@pytest.mark.parametrize("keep_registers", [True, False])
def test_registers_are_never_candidates(keep_registers):
    b = tiny_batch(B=2, segs=3, P=(6, 5), R=3, M=(2, 3), seed=14)
    out = O.prune(b, 0.0, 0.0, keep_registers=keep_registers)
    is_reg = out["is_reg"]
    assert out["count_vis"].sum() == (~is_reg).sum()
    assert bool(np.isin(np.nonzero(is_reg)[0], out["out_index"]).all()) == keep_registers
    assert not np.isin(np.nonzero(is_reg)[0], out["out_index"]).any() or keep_registers
    assert out["count_out"].sum() == (~is_reg).sum() + (is_reg.sum() if keep_registers else 0)


# ----------------------------------------------------------------------------- P13 scale invariance

def test_threshold_scale_invariant():
    rng = np.random.default_rng(2)
    s = rng.random(100)
    ref = np.full(100, 0.4)
    is_reg = np.zeros(100, bool)
    is_reg[[3, 50]] = True
    base = O.threshold(s, ref, 1.3, is_reg)
    for c in (1e-3, 0.5, 7.0):
        assert (O.threshold(s * c, ref * c, 1.3, is_reg) == base).all()


# ----------------------------------------------------------------------------- P11 brute force

def _dexp(x):
    return x.exp()


def _brute_stage1_cls(q, kc, K, seg_off, reg_idx, reg_off):
    H, d = len(K[0]), len(K[0][0])
    sc = Decimal(1) / Decimal(d).sqrt()
    s1 = [Decimal(0)] * len(K)
    ref = []
    for s in range(len(seg_off) - 1):
        rows = range(seg_off[s], seg_off[s + 1])
        for h in range(H):
            dot = lambda a, b: sum(Decimal(x) * Decimal(y) for x, y in zip(a, b))  # noqa: E731
            logits = {r: dot(q[s][h], K[r][h]) * sc for r in rows}
            z = sum(_dexp(v) for v in logits.values())
            if kc is not None:
                z += _dexp(dot(q[s][h], kc[s][h]) * sc)
            for r in rows:
                s1[r] += _dexp(logits[r]) / z / H
        regs = reg_idx[reg_off[s]:reg_off[s + 1]]
        ref.append(sum(s1[r] for r in regs) / len(regs))
    return s1, ref


def _brute_stage1_mutual(Q, K, seg_off, reg_idx, reg_off):
    H, d = len(K[0]), len(K[0][0])
    sc = Decimal(1) / Decimal(d).sqrt()
    s1 = [Decimal(0)] * len(K)
    ref = []
    dot = lambda a, b: sum(Decimal(x) * Decimal(y) for x, y in zip(a, b))  # noqa: E731
    for s in range(len(seg_off) - 1):
        rows = list(range(seg_off[s], seg_off[s + 1]))
        n = len(rows)
        for h in range(H):
            for u in rows:
                e = {v: _dexp(dot(Q[u][h], K[v][h]) * sc) for v in rows}
                z = sum(e.values())
                for v in rows:
                    s1[v] += e[v] / z / H / n
        regs = reg_idx[reg_off[s]:reg_off[s + 1]]
        ref.append(sum(s1[r] for r in regs) / len(regs))
    return s1, ref


def _brute_stage2(Q, Kt, K, keep1, is_reg, row_off, text_off):
    H, d = len(K[0]), len(K[0][0])
    sc = Decimal(1) / Decimal(d).sqrt()
    dot = lambda a, b: sum(Decimal(x) * Decimal(y) for x, y in zip(a, b))  # noqa: E731
    s2 = [Decimal(0)] * len(K)
    ref2 = []
    for b in range(len(row_off) - 1):
        S1 = [r for r in range(row_off[b], row_off[b + 1]) if keep1[r] or is_reg[r]]
        texts = list(range(text_off[b], text_off[b + 1]))
        M = len(texts)
        regsum = Decimal(0)
        regs = [r for r in S1 if is_reg[r]]
        best = {r: Decimal(0) for r in S1}
        for jj, j in enumerate(texts):
            p = {r: Decimal(0) for r in S1}
            for h in range(H):
                e = {r: _dexp(dot(Q[j][h], K[r][h]) * sc) for r in S1}
                z = sum(e.values()) + sum(_dexp(dot(Q[j][h], Kt[t][h]) * sc) for t in texts[:jj + 1])
                for r in S1:
                    p[r] += e[r] / z / H
            for r in S1:
                best[r] = max(best[r], p[r])
            regsum += sum(p[r] for r in regs) / len(regs)
        for r in S1:
            if not is_reg[r]:
                s2[r] = best[r]
        ref2.append(regsum / M)
    return s2, ref2


def _lists(t):
    return t.float().tolist()


def test_brute_force_decimal_tiny():
    """Every score recomputed with 50-digit decimals; all lambda breakpoints checked."""
    getcontext().prec = 50
    b = tiny_batch(B=2, segs=2, P=(3, 4), R=1, M=(2, 3), H1=2, d1=4, H2=2, d2=4, seed=15)
    m = b["meta"]
    out = O.prune(b, 0.9, 1.0)
    s1, ref1 = _brute_stage1_cls(_lists(b["q_cls"]), _lists(b["k_cls"]), _lists(b["K1"]),
                                 m["seg_off_host"].tolist(), m["reg_idx_host"].tolist(), m["reg_off_host"].tolist())
    np.testing.assert_allclose(out["s1"], [float(x) for x in s1], rtol=1e-14)
    np.testing.assert_allclose(out["ref1"], [float(x) for x in ref1], rtol=1e-14)
    is_reg = out["is_reg"]
    s2, ref2 = _brute_stage2(_lists(b["Q_text"]), _lists(b["K_text"]), _lists(b["K2"]), out["keep1"].tolist(),
                             is_reg.tolist(), m["row_off_host"].tolist(), m["text_off_host"].tolist())
    np.testing.assert_allclose(out["s2"], [float(x) for x in s2], rtol=1e-14, atol=0)
    np.testing.assert_allclose(out["ref2"], [float(x) for x in ref2], rtol=1e-14)
    # Stage-I count as a step function of lambda1: it drops exactly at each ratio
    seg_of_row = np.repeat(np.arange(m["S_tot"]), np.diff(m["seg_off_host"]))
    ratios = sorted(float(s1[r] / ref1[seg_of_row[r]]) for r in range(m["total_rows"]) if not is_reg[r])
    for i, x in enumerate(ratios):
        n_at = O.prune(b, x * (1 - 1e-12), 0.0)["n1_vis"].sum()
        n_after = O.prune(b, x * (1 + 1e-12), 0.0)["n1_vis"].sum()
        assert n_at == len(ratios) - i and n_after == len(ratios) - i - 1


def test_brute_force_decimal_mutual():
    getcontext().prec = 50
    b = tiny_batch(B=2, segs=1, P=(4, 3), R=2, M=(2, 2), H1=2, d1=4, stage1="mutual", seed=16)
    m = b["meta"]
    s1, ref1 = O.stage1_mutual(b["Q1"], b["K1"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"])
    bs1, bref = _brute_stage1_mutual(_lists(b["Q1"]), _lists(b["K1"]), m["seg_off_host"].tolist(),
                                     m["reg_idx_host"].tolist(), m["reg_off_host"].tolist())
    np.testing.assert_allclose(s1, [float(x) for x in bs1], rtol=1e-14)
    np.testing.assert_allclose(ref1, [float(x) for x in bref], rtol=1e-14)


def test_head_reduce_reading_differs_from_alternative():
    """The 'max over (text, head)' reading is a different function (flag works)."""
    b = tiny_batch(B=1, segs=2, P=(8,), R=2, M=(5,), H2=4, seed=17)
    a = O.prune(b, 0.0, 1.0)
    c = O.prune(b, 0.0, 1.0, head_reduce="max")
    vis = ~a["is_reg"]
    assert (c["s2"][vis] >= a["s2"][vis] - 1e-15).all()
    assert (c["s2"][vis] > a["s2"][vis] * (1 + 1e-6)).any()


# ----------------------------------------------------------------------------- n_eff (Sec. 3.2, Observation 1)

def test_neff_uniform_attention_counts_every_key():
    """q_cls = 0: the [CLS] attention is uniform over the N keys ({[CLS]} u rows), so n_eff = N."""
    b = tiny_batch(B=2, segs=2, P=(5, 8), R=3, M=(2, 3), seed=6)
    m = b["meta"]
    ne = O.stage1_neff(_zero(b["q_cls"]), b["k_cls"], b["K1"], m["seg_off_host"])
    n_keys = np.diff(m["seg_off_host"]) + 1
    np.testing.assert_allclose(ne, np.repeat(n_keys[:, None], ne.shape[1], axis=1), rtol=1e-13)
    # without the [CLS] key, the rows alone
    ne2 = O.stage1_neff(_zero(b["q_cls"]), None, b["K1"], m["seg_off_host"])
    np.testing.assert_allclose(ne2[:, 0], n_keys - 1, rtol=1e-13)


@pytest.mark.parametrize("dl", [0, 1, 3, 40])
def test_neff_two_keys_binary_entropy(dl):
    """Two keys with an exact logit gap dl: a = (p, 1-p), p = 1/(1+e^-dl), n_eff = exp(h(p))."""
    q = torch.tensor([[[2.0, 0, 0, 0]]]).to(torch.bfloat16)          # scale 1/2 -> logit = k[0]
    K1 = torch.tensor([[[float(dl), 1, 2, 3]], [[0.0, -1, 5, 2]]]).to(torch.bfloat16)
    ne = O.stage1_neff(q, None, K1, np.array([0, 2]))
    p = 1.0 / (1.0 + math.exp(-dl))
    h = -(p * math.log(p) + (1 - p) * math.log1p(-p)) if p < 1 else 0.0
    assert abs(ne[0, 0] - math.exp(h)) <= 1e-12 * math.exp(h)
    assert 1.0 <= ne[0, 0] <= 2.0 + 1e-15
    if dl == 0:
        assert abs(ne[0, 0] - 2.0) < 1e-14


def test_neff_bounds_and_heads_independent():
    """1 <= n_eff <= N on random inputs; identical heads give identical values."""
    b = tiny_batch(B=2, segs=2, P=(9, 14), R=2, M=(2, 2), seed=31)
    m = b["meta"]
    ne = O.stage1_neff(b["q_cls"], b["k_cls"], b["K1"], m["seg_off_host"])
    n_keys = np.diff(m["seg_off_host"]) + 1
    assert (ne >= 1.0 - 1e-12).all() and (ne <= n_keys[:, None] + 1e-9).all()
    q = b["q_cls"].clone()
    K = b["K1"].clone()
    q[:] = q[:, :1]
    K[:] = K[:, :1]
    ne_same = O.stage1_neff(q, b["k_cls"][:, :1].expand_as(b["k_cls"]).contiguous(), K, m["seg_off_host"])
    assert np.all(ne_same == ne_same[:, :1])


def test_neff_brute_force_decimal_tiny():
    """exp(-sum a log a) at 50 digits from the exact bf16 values."""
    getcontext().prec = 50
    b = tiny_batch(B=1, segs=2, P=(3,), R=1, M=(2,), H1=2, d1=4, seed=33)
    m = b["meta"]
    ne = O.stage1_neff(b["q_cls"], b["k_cls"], b["K1"], m["seg_off_host"])
    q = O.as_f64(b["q_cls"])
    kc = O.as_f64(b["k_cls"])
    K = O.as_f64(b["K1"])
    sc = Decimal(1) / Decimal(4).sqrt()
    dot = lambda a, c: sum(Decimal(float(x)) * Decimal(float(y)) for x, y in zip(a, c))  # noqa: E731
    so = m["seg_off_host"]
    for s in range(len(so) - 1):
        for h in range(2):
            lg = [dot(kc[s, h], q[s, h]) * sc] + [dot(K[r, h], q[s, h]) * sc for r in range(so[s], so[s + 1])]
            mx = max(lg)
            e = [(x - mx).exp() for x in lg]
            z = sum(e)
            a = [x / z for x in e]
            want = (-sum(x * x.ln() for x in a)).exp()
            assert abs(Decimal(ne[s, h]) - want) <= Decimal("1e-12") * want


# ----------------------------------------------------------------------------- lambda2 budget matching (App. A)

def _ratio_count(s2, ref2, keep1, is_reg, row_off, lam):
    """Rows the Stage-II test keeps at lam, as the library applies it: s2 >= fl(lam * ref2) in fp32
    (visual S1 rows of samples with a positive reference), one row at a time."""
    s2 = np.asarray(s2, np.float32)
    ref2 = np.asarray(ref2, np.float32)
    n = 0
    for b in range(len(row_off) - 1):
        if not ref2[b] > 0:
            continue
        tau = np.float32(lam) * ref2[b]
        for v in range(row_off[b], row_off[b + 1]):
            n += int(bool(keep1[v]) and not is_reg[v] and s2[v] >= tau)
    return n


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_lambda2_budget_is_the_count_step(seed):
    """At lambda2* the ratio test keeps >= K rows, just above it < K; every K of a small set, brute force."""
    rng = np.random.default_rng(seed)
    row_off = np.array([0, 7, 7, 19, 30])
    R = row_off[-1]
    s2 = rng.random(R).astype(np.float32) * rng.choice([1e-3, 1.0], R).astype(np.float32)
    ref2 = np.array([0.2, 0.5, 0.01, 0.0], np.float32)       # the last sample has no positive reference
    keep1 = rng.random(R) < 0.7
    is_reg = np.zeros(R, bool)
    is_reg[[6, 18]] = True
    n = _ratio_count(s2, ref2, keep1, is_reg, row_off, 0.0)
    for K in range(0, n + 2):
        lam, cnt = O.lambda2_for_budget(s2, ref2, keep1, is_reg, row_off, K)
        assert cnt == n
        if K == 0:
            assert np.isinf(lam)
            continue
        if K > n:
            assert lam == 0.0
            continue
        assert _ratio_count(s2, ref2, keep1, is_reg, row_off, lam) >= K
        assert _ratio_count(s2, ref2, keep1, is_reg, row_off, np.nextafter(lam, np.float32(np.inf))) < K


def test_lambda2_budget_on_oracle_scores_matches_the_threshold_rule():
    """On oracle Stage-II scores, lambda2* of a budget gives that budget through O.threshold."""
    b = tiny_batch(B=3, segs=2, P=(20, 13, 31), R=2, M=(5, 9, 2), seed=10)
    out = O.prune(b, 0.9, 1.2)
    m = b["meta"]
    row_off = m["row_off_host"]
    n_vis1 = int(np.sum(out["keep1"] & ~out["is_reg"]))
    sample = np.repeat(np.arange(m["B"]), np.diff(row_off))
    s2f = np.asarray(out["s2"], np.float32)
    r2f = np.asarray(out["ref2"], np.float32)
    for K in (1, n_vis1 // 3, n_vis1 - 1):
        lam, _ = O.lambda2_for_budget(s2f, r2f, out["keep1"], out["is_reg"], row_off, K)
        # the rule with lambda2 applied as one fp32 product keeps at least K rows, and fewer one step up
        keep = out["keep1"] & ~out["is_reg"] & (s2f >= np.float32(lam) * r2f[sample])
        keep_up = out["keep1"] & ~out["is_reg"] & (s2f >= np.nextafter(lam, np.float32(np.inf)) * r2f[sample])
        assert int(keep.sum()) >= K > int(keep_up.sum())


def test_lambda2_budget_product_rounding():
    """The defining row survives the product test: for every candidate v of random fp32 pairs, the
    budget that ends at v's quotient keeps v (the quotient alone rounds up in a few percent of pairs)."""
    rng = np.random.default_rng(7)
    n = 4000
    s2 = rng.random(n).astype(np.float32) * np.float32(1e-3)
    ref2 = np.array([np.float32(0.0123457)], np.float32)
    row_off = np.array([0, n])
    keep1 = np.ones(n, bool)
    is_reg = np.zeros(n, bool)
    order = np.argsort(-(s2 / ref2[0]), kind="stable")
    bad_quotients = 0
    for K in range(1, n + 1, 37):
        v = order[K - 1]
        q = s2[v] / ref2[0]
        bad_quotients += int(not (s2[v] >= q * ref2[0]))
        lam, _ = O.lambda2_for_budget(s2, ref2, keep1, is_reg, row_off, K)
        assert s2[v] >= np.float32(lam) * ref2[0]
        assert int(np.sum(s2 >= np.float32(lam) * ref2[0])) >= K
    assert bad_quotients > 0  # the case the stepping exists for does occur


# ----------------------------------------------------------------------------- register construction (Algorithm 1)

def test_register_construction_properties():
    """Per segment and register channel: the registers hold a value that bounds every visual entry and
    equals one of them; the visual entries are 0; every other entry is untouched; the result does not
    depend on the order of the visual rows."""
    b = tiny_batch(B=2, segs=3, P=(9, 14), R=2, M=(2, 2), hidden=32, seed=61)
    m = b["meta"]
    h = b["hidden"].clone()
    h[3, 5] = 40.0                                           # a sink-like activation
    k_reg = np.array([5, 17, 30])
    out = O.construct_registers(h, m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"], k_reg)
    before = O.as_f64(h)
    so, ri, ro = m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"]
    other = np.setdiff1d(np.arange(before.shape[1]), k_reg)
    assert np.array_equal(out[:, other], before[:, other])
    for s in range(m["S_tot"]):
        regs = ri[ro[s]:ro[s + 1]]
        vis = np.setdiff1d(np.arange(so[s], so[s + 1]), regs)
        for k in k_reg:
            v = before[vis, k]
            for r in regs:
                assert all(out[r, k] >= x for x in v) and any(out[r, k] == x for x in v)
            assert np.all(out[vis, k] == 0.0)
    assert out[ri[ro[0]], 5] == 40.0 or 3 not in range(so[0], so[1])
    # permuting the visual rows of a segment changes nothing at the registers
    perm = before.copy()
    vis0 = np.setdiff1d(np.arange(so[0], so[1]), ri[ro[0]:ro[1]])
    perm[vis0] = perm[vis0[::-1]]
    out2 = O.construct_registers(torch.from_numpy(perm), so, ri, ro, k_reg)
    assert np.array_equal(out2[ri[ro[0]:ro[1]]][:, k_reg], out[ri[ro[0]:ro[1]]][:, k_reg])


# ----------------------------------------------------------------------------- rule variants (component ablation)

def test_mean_reference_hand_values():
    """Mean over the unit's candidates only (registers and rows outside prev_keep excluded); 0 without any."""
    s = np.array([1.0, 2.0, 6.0, 100.0, 5.0, 7.0, 3.0])
    is_reg = np.array([False, False, False, True, False, False, True])
    prev = np.array([True, True, True, True, False, True, True])
    ref = O.mean_reference(s, np.array([0, 4, 7]), ~is_reg)
    assert ref.tolist() == [3.0, 6.0]
    ref = O.mean_reference(s, np.array([0, 4, 7]), ~is_reg & prev)
    assert ref.tolist() == [3.0, 7.0]
    ref = O.mean_reference(s, np.array([0, 3, 4, 7]), ~is_reg & prev)
    assert ref.tolist() == [3.0, 0.0, 7.0]                   # the middle unit holds only a register


def _budget_brute(s, rows, k):
    """The unique k-subset of `rows` whose every member precedes every non-member in the
    order (score high first, row low first), by enumeration."""
    import itertools
    found = []
    for sub in itertools.combinations(rows, k):
        rest = [r for r in rows if r not in sub]
        if all((s[a] > s[d]) or (s[a] == s[d] and a < d) for a in sub for d in rest):
            found.append(set(sub))
    assert len(found) == 1
    return found[0]


@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_budget_keep_brute_force(seed):
    """Fixed budget = the top-K rule of Sec. 2 with ties taken lower row first; brute force over subsets."""
    rng = np.random.default_rng(seed)
    row_off = np.array([0, 8, 8, 15, 22])
    R = row_off[-1]
    s = rng.choice([0.0, 0.1, 0.2, 0.3, 0.5], R)             # many ties
    is_reg = np.zeros(R, bool)
    is_reg[[7, 14]] = True
    cand = rng.random(R) < 0.8
    budget = np.array([3, 2, 9, 0])
    keep, count = O.budget_keep(s, row_off, cand, budget, is_reg, keep_registers=True)
    for b in range(4):
        rows = [r for r in range(row_off[b], row_off[b + 1]) if cand[r] and not is_reg[r]]
        k = min(budget[b], len(rows))
        assert count[b] == k
        want = _budget_brute(s, rows, k) if rows else set()
        got = {r for r in range(row_off[b], row_off[b + 1]) if keep[r] and not is_reg[r]}
        assert got == want
    assert keep[is_reg].all()
    keep0, _ = O.budget_keep(s, row_off, cand, budget, is_reg, keep_registers=False)
    assert not keep0[is_reg].any()


def test_budget_rule_equals_the_method_at_its_own_counts():
    """With budget[b] = the method's count_vis the fixed-budget rule keeps the same rows (the threshold
    keeps the top count_vis of s2 per sample; no ties at the threshold in these inputs)."""
    b = tiny_batch(B=3, segs=2, P=(20, 13, 31), R=2, M=(5, 9, 2), seed=10)
    ref = O.prune(b, 0.9, 1.2)
    bud = O.prune(b, 0.9, 1.2, rule="budget", budget=ref["count_vis"])
    assert np.array_equal(bud["keep1"], ref["keep1"])
    assert np.array_equal(bud["keep2"], ref["keep2"])
    half = O.prune(b, 0.9, 1.2, rule="budget", budget=ref["count_vis"] // 2)
    assert np.array_equal(half["count_vis"], ref["count_vis"] // 2)
    assert not (half["keep2"] & ~ref["keep2"]).any()           # a smaller budget keeps a subset


def test_mean_rule_equals_the_method_at_a_matched_lambda():
    """One segment, one sample: the mean rule at lambda * s(r) / mean gives the method's threshold, so the
    same sets (rows within 1e-9 of either threshold are avoided)."""
    b = tiny_batch(B=1, segs=1, P=(40,), R=2, M=(6,), seed=21)
    lam1, lam2 = 0.9, 1.1
    ref = O.prune(b, lam1, lam2)
    is_reg = ref["is_reg"]
    m1 = O.mean_reference(ref["s1"], b["meta"]["seg_off_host"], ~is_reg)[0]
    m2 = O.mean_reference(ref["s2"], b["meta"]["row_off_host"], ref["keep1"] & ~is_reg)[0]
    mean = O.prune(b, lam1 * ref["ref1"][0] / m1, lam2 * ref["ref2"][0] / m2, rule="mean")
    assert np.isclose(mean["ref1"][0], m1) and np.isclose(mean["ref2"][0], m2)
    assert np.allclose(mean["tau1"], ref["tau1"], rtol=1e-12)
    assert np.allclose(mean["tau2"], ref["tau2"], rtol=1e-12)
    assert np.min(np.abs(ref["s1"] - ref["tau1"])[~is_reg]) > 1e-9 * ref["tau1"][0]
    assert np.array_equal(mean["keep1"], ref["keep1"])
    assert np.array_equal(mean["keep2"], ref["keep2"])
    # the mean of the visual scores differs from the register reference: the rule is not a no-op
    assert abs(m1 - ref["ref1"][0]) > 1e-3 * m1


# ----------------------------------------------------------------------------- grouped-query Stage II

@pytest.mark.parametrize("text_keys", ["causal", "none"])
def test_grouped_query_heads_equal_expanded_keys(text_keys):
    """H_kv key heads shared by groups of H / H_kv query heads = H separate heads whose keys are copies
    (query head h reading key head h // group). A wrong group index (h % H_kv) fails this."""
    b = tiny_batch(B=2, segs=2, P=(9, 14), R=2, M=(5, 7), H2=8, H2kv=2, d2=16, seed=91)
    assert b["K2"].shape[1] == 2 and b["Q_text"].shape[1] == 8
    full = dict(b)
    idx = torch.arange(8) // 4
    full["K2"] = b["K2"][:, idx, :].contiguous()
    full["K_text"] = b["K_text"][:, idx, :].contiguous()
    g = O.prune(b, 0.6, 1.1, text_keys=text_keys)
    e = O.prune(full, 0.6, 1.1, text_keys=text_keys)
    assert np.array_equal(g["s2"], e["s2"]) and np.array_equal(g["ref2"], e["ref2"])
    assert np.array_equal(g["keep2"], e["keep2"])
    # and the grouping matters: pairing query head h with key head h % H_kv gives other scores
    wrong = dict(b)
    wrong["K2"] = b["K2"][:, torch.arange(8) % 2, :].contiguous()
    wrong["K_text"] = b["K_text"][:, torch.arange(8) % 2, :].contiguous()
    assert not np.allclose(O.prune(wrong, 0.6, 1.1, text_keys=text_keys)["s2"], g["s2"])


# ----------------------------------------------------------------------------- merged-token pooling (Qwen 2x2 merger)

def test_pool_scores_hand_values_and_mass():
    s = np.array([0.1, 0.2, 0.3, 0.4, 1.0, 0.0, 0.0, 3.0])
    assert np.allclose(O.pool_scores(s, 4, "sum"), [1.0, 4.0])
    assert np.allclose(O.pool_scores(s, 4, "mean"), [0.25, 1.0])
    assert O.pool_scores(s, 4, "max").tolist() == [0.4, 3.0]
    assert O.pool_scores(s, 1, "sum").tolist() == s.tolist()
    # sum pooling keeps the total attention mass of a segment's [CLS] row
    b = tiny_batch(B=1, segs=1, P=(38,), R=2, M=(2,), seed=5, H1=4, d1=16)
    s1, _ = O.stage1_cls(b["q_cls"], None, b["K1"], b["meta"]["seg_off_host"], b["meta"]["reg_idx_host"],
                         b["meta"]["reg_off_host"])
    assert abs(O.pool_scores(s1, 4, "sum").sum() - 1.0) < 1e-12
    with pytest.raises(AssertionError):
        O.pool_scores(np.zeros(6), 4)
