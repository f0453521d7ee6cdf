"""CPU oracle for the OccamToken prune path (test infrastructure only).

This module is the plain, slow definition that the CUDA path is checked
against. Only the tests, the smoke check and the bench's CPU-baseline leg use
it; the product path never imports, links or calls anything here.

Everything is computed in float64 from the exact values of the bf16 inputs.
Each function follows one equation of the paper:

* scaled dot-product attention, A = softmax(Q K^T / sqrt(d_h))   -- Sec. 3.1, Eq. 1
* relative comparison rule s_x(v) >= lambda s_x(r(x))            -- Sec. 3.2, Eq. 3
* Stage I [CLS] scores s1(v) = A_{cls->v}, s1(r) = A_{cls->r},
  averaged over heads                                            -- Sec. 3.4, Eq. 4; App. A, Eq. 10
* effective number of attended keys n_eff = exp(H(A)) of the
  Stage-I [CLS] attention, per segment and head                 -- Sec. 3.2, Observation 1
* Stage I mutual scores s1(v) = 1/(|V|+1) sum_u A_{u->v}         -- Sec. 3.4, Eq. 6; App. A, Eq. 13
* Stage I set S1 = {v : s1(v) >= lambda1 s1(r)} u {r}            -- Eq. 5; App. A, Eqs. 11-12
* Stage II scores s2(v) = max_j A_{t_j->v}, s2(r) = mean_j A_{t_j->r}
                                                                 -- Sec. 3.5, Eq. 7; App. A, Eqs. 15-16
* Stage II set S2 = {v in S1\\{r} : s2(v) >= lambda2 s2(r)} u {r} -- Eq. 8; App. A, Eq. 17
* lambda2 matching a retained budget over a calibration set      -- App. A, average-budget equation
* test-time register construction h_r,k = max_v h_v,k, h_v,k = 0 -- Algorithm 1; App. A, register redirection
* pooling of patch scores onto merged tokens (Qwen3-VL's 2x2 patch merger
  puts each merged token's four patches on consecutive rows)   -- Sec. 4 setup; reading below
* rule variants of the component ablation (App., "compact component
  ablation"): a mean-based reference instead of the register's score, and a
  fixed per-sample budget (the top-K rule of Sec. 2) instead of the
  Stage-II threshold                                             -- Sec. 2, top-K rule; ablation table
* decoding continues on [S2; T]: order-preserving compaction of
  the kept rows (prefix and KV cache shrink with the kept count) -- Algorithm 1; App. A, Eq. 21

Readings where the paper is silent (each one is also a keyword flag here):

* heads: per-head probabilities are averaged over heads before the max / mean
  over text tokens (App. A says the vision map is "averaged over attention
  heads"; the LLM map is read the same way). ``stage2_head_reduce="max"``
  takes the max over (text token, head) instead;
* several registers per segment (the paper has one): the reference score is
  the mean of the registers' scores -- over the segment's registers in
  Stage I, over all of the sample's registers in Stage II;
* multi-crop / multi-frame samples: Stage I runs per segment (each crop or
  frame has its own [CLS] query, softmax, registers and threshold); Stage II
  runs per sample over the union of the segments' survivors;
* the [CLS] token's own key is part of the Stage-I softmax when ``k_cls`` is
  given; [CLS] itself is never a candidate;
* the Stage-II softmax of text token j runs over the S1 rows (visual
  survivors and every register, image first) and the text keys 0..j
  (causal); ``text_keys="none"`` drops the text keys;
* the mutual-mode average divides by the segment's row count P+R;
* ties keep (the test is >=); lambda <= 0 keeps every visual row;
* the mean threshold takes, per stage, the mean score of that stage's
  candidates (Stage I: the segment's visual rows; Stage II: the sample's
  visual S1 rows) as the reference, in both stages;
* merged tokens (the paper is silent on how patch scores become merged-token
  scores): the score of a group of consecutive patch rows is the sum of its
  patches' scores (the attention mass the merged token receives); the mean
  and the max are flags;
* the fixed budget keeps Stage I as in the method and, per sample, the
  budget[b] visual S1 rows with the largest s2 (all of them when there are
  fewer); equal scores keep the lower row first;
* kept rows are emitted in ascending row order, samples in batch order.

Parity pins live in tests/test_oracle_pins.py; no function here is
"parity unpinned".
"""

from __future__ import annotations

import numpy as np


def as_f64(x) -> np.ndarray:
    """Exact float64 copy of a bf16/fp32 array (bf16 -> fp32 -> fp64 is exact)."""
    if hasattr(x, "detach"):  # torch tensor
        import torch
        x = x.detach().to("cpu")
        if x.dtype == torch.bfloat16:
            x = x.to(torch.float32)
        x = x.numpy()
    return np.asarray(x, dtype=np.float64)


def as_i64(x) -> np.ndarray:
    if hasattr(x, "detach"):
        x = x.detach().to("cpu").numpy()
    return np.asarray(x, dtype=np.int64)


def softmax(logits: np.ndarray, axis: int = -1) -> np.ndarray:
    """Softmax along ``axis`` (Sec. 3.1, Eq. 1): exp(l - max) / sum(exp(l - max))."""
    m = np.max(logits, axis=axis, keepdims=True)
    e = np.exp(logits - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def register_mask(total_rows: int, reg_idx) -> np.ndarray:
    mask = np.zeros(total_rows, dtype=bool)
    mask[as_i64(reg_idx)] = True
    return mask


# --------------------------------------------------------------------------- Stage I

def stage1_cls(q_cls, k_cls, K1, seg_off, reg_idx, reg_off):
    """Stage-I [CLS] scores (Sec. 3.4, Eq. 4; App. A, Eq. 10 with its head average).

    For each segment s and head h the [CLS] query of s attends to the keys
    {k_cls[s]} u rows(s) with A = softmax(q k^T / sqrt(d1)); s1[row] is the
    mean over heads of A_h(row); ref1[s] is the mean of s1 over the segment's
    registers. Returns (s1 [rows], ref1 [S_tot]).
    """
    q = as_f64(q_cls)
    kc = None if k_cls is None else as_f64(k_cls)
    K = as_f64(K1)
    seg_off = as_i64(seg_off)
    reg_idx = as_i64(reg_idx)
    reg_off = as_i64(reg_off)
    S_tot = seg_off.shape[0] - 1
    H, d = K.shape[1], K.shape[2]
    scale = 1.0 / np.sqrt(d)
    s1 = np.zeros(K.shape[0], dtype=np.float64)
    ref1 = np.zeros(S_tot, dtype=np.float64)
    for s in range(S_tot):
        r0, r1 = seg_off[s], seg_off[s + 1]
        for h in range(H):
            logits_rows = (K[r0:r1, h, :] @ q[s, h, :]) * scale
            if kc is not None:
                logit_cls = np.dot(kc[s, h, :], q[s, h, :]) * scale
                A = softmax(np.concatenate([[logit_cls], logits_rows]))[1:]
            else:
                A = softmax(logits_rows)
            s1[r0:r1] += A / H
        regs = reg_idx[reg_off[s]:reg_off[s + 1]]
        ref1[s] = np.mean(s1[regs])
    return s1, ref1


def effective_keys(a) -> float:
    """n_eff = exp(H(a)) with H(a) = -sum_i a_i log a_i, the entropy of an
    attention distribution a (Sec. 3.2, Observation 1): the support size of
    the uniform distribution with the same entropy. Terms with a_i = 0 add 0."""
    a = np.asarray(a, dtype=np.float64)
    terms = np.where(a > 0, a * np.log(np.where(a > 0, a, 1.0)), 0.0)
    return float(np.exp(-np.sum(terms)))


def stage1_neff(q_cls, k_cls, K1, seg_off):
    """n_eff of the Stage-I [CLS] attention (Sec. 3.2, Observation 1, on the
    map of Sec. 3.4, Eq. 4): for each segment s and head h, the distribution
    A = softmax(q k^T / sqrt(d1)) of the segment's [CLS] query over the keys
    {k_cls[s]} u rows(s) (the [CLS] key included when given), and
    n_eff = exp(-sum A log A). Returns [S_tot, H].
    """
    q = as_f64(q_cls)
    kc = None if k_cls is None else as_f64(k_cls)
    K = as_f64(K1)
    seg_off = as_i64(seg_off)
    S_tot = seg_off.shape[0] - 1
    H, d = K.shape[1], K.shape[2]
    scale = 1.0 / np.sqrt(d)
    out = np.zeros((S_tot, H), dtype=np.float64)
    for s in range(S_tot):
        r0, r1 = seg_off[s], seg_off[s + 1]
        for h in range(H):
            logits = (K[r0:r1, h, :] @ q[s, h, :]) * scale
            if kc is not None:
                logits = np.concatenate([[np.dot(kc[s, h, :], q[s, h, :]) * scale], logits])
            out[s, h] = effective_keys(softmax(logits))
    return out


def stage1_mutual(Q1, K1, seg_off, reg_idx, reg_off):
    """Stage-I mutual scores (Sec. 3.4, Eq. 6; App. A, Eq. 13).

    Within segment s every row u (visual or register) attends to every row v
    of s, per head; s1[v] = 1/(P+R) * sum_u mean_h A_h(u -> v); ref1[s] is the
    mean of s1 over the segment's registers.
    """
    Q = as_f64(Q1)
    K = as_f64(K1)
    seg_off = as_i64(seg_off)
    reg_idx = as_i64(reg_idx)
    reg_off = as_i64(reg_off)
    S_tot = seg_off.shape[0] - 1
    H, d = K.shape[1], K.shape[2]
    scale = 1.0 / np.sqrt(d)
    s1 = np.zeros(K.shape[0], dtype=np.float64)
    ref1 = np.zeros(S_tot, dtype=np.float64)
    for s in range(S_tot):
        r0, r1 = seg_off[s], seg_off[s + 1]
        n = r1 - r0
        acc = np.zeros(n, dtype=np.float64)
        for h in range(H):
            A = softmax((Q[r0:r1, h, :] @ K[r0:r1, h, :].T) * scale, axis=1)  # [u, v]
            acc += A.sum(axis=0) / H
        s1[r0:r1] = acc / n
        regs = reg_idx[reg_off[s]:reg_off[s + 1]]
        ref1[s] = np.mean(s1[regs])
    return s1, ref1


# --------------------------------------------------------------------------- thresholds

def threshold(s, ref_of_row, lam: float, is_reg, prev_keep=None, keep_registers: bool = True):
    """Register-anchored test s(v) >= lambda * s(r) (Eq. 3; Stage I Eq. 5, Stage II Eq. 8).

    Visual rows are candidates; a row passes when its score is at least
    ``lam`` times its reference (``ref_of_row``, already broadcast per row);
    ``prev_keep`` restricts the candidates (Stage II only looks at S1).
    Register rows are not candidates; they are kept iff ``keep_registers``.
    Scores are probabilities (>= 0), so ``lam <= 0`` keeps every candidate
    (Table 5: lambda1 = 0 is "w/o Stage I").
    """
    s = np.asarray(s, dtype=np.float64)
    tau = float(lam) * np.asarray(ref_of_row, dtype=np.float64)
    keep = s >= tau
    if prev_keep is not None:
        keep &= np.asarray(prev_keep, dtype=bool)
    keep &= ~is_reg
    if keep_registers:
        keep |= is_reg
    return keep


def construct_registers(h, seg_off, reg_idx, reg_off, k_reg):
    """Test-time register construction (Algorithm 1, step 2; App. A, register
    redirection): for every segment and register channel k, each register
    row takes the max of channel k over the segment's visual rows, and the
    channel is then zeroed on those visual rows. A segment without visual
    rows keeps its registers. Returns a new float64 array (the bf16 inputs
    are exact in it; the results are inputs or 0, so exact in bf16 too).
    """
    h = as_f64(h).copy()
    seg_off = as_i64(seg_off)
    reg_idx = as_i64(reg_idx)
    reg_off = as_i64(reg_off)
    for s in range(len(seg_off) - 1):
        rows = np.arange(seg_off[s], seg_off[s + 1])
        regs = reg_idx[reg_off[s]:reg_off[s + 1]]
        vis = np.setdiff1d(rows, regs)
        for k in as_i64(k_reg):
            if len(vis) > 0:
                h[regs, k] = np.max(h[vis, k])
                h[vis, k] = 0.0
    return h


def lambda2_for_budget(s2, ref2, keep1, is_reg, row_off, target_count: int):
    """lambda2 matching a retained budget (App. A, the lambda2* that makes the
    average |S2| over the calibration set D equal K_tar).

    |S2(lambda2)| counts the visual S1 rows v with s2(v) >= lambda2 s2(r) of
    their sample, so the total over D drops by one at each ratio
    s2(v) / s2(r). The lambda2 whose total is K = target_count
    (= K_tar |D|) is therefore the K-th largest ratio. The scores are fp32,
    and the rule applies lambda2 as one fp32 product (s2(v) >= fl(lambda2
    s2(r))), so lambda2* is taken as the largest fp32 value under which that
    product test keeps at least K rows: the K-th largest fp32 quotient
    s2(v) / s2(r) (from a sort), moved by single fp32 steps while the
    product's rounding disagrees with the quotient's (a few ulps at most).
    Just above lambda2* the test keeps fewer than K rows. Samples whose
    reference is not positive contribute no candidates. K <= 0 gives +inf;
    K above the candidate count gives 0 (keep all).
    """
    s2 = np.asarray(s2, dtype=np.float32)
    ref2 = np.asarray(ref2, dtype=np.float32)
    row_off = as_i64(row_off)
    cand = np.asarray(keep1, dtype=bool) & ~np.asarray(is_reg, dtype=bool)
    sample = np.repeat(np.arange(len(row_off) - 1), np.diff(row_off))
    cand &= ref2[sample] > 0
    s2c, refc = s2[cand], ref2[sample][cand]
    ratios = np.sort(s2c / refc)[::-1]  # float32 / float32: IEEE quotient
    if target_count <= 0:
        return np.float32(np.inf), int(cand.sum())
    if target_count > len(ratios):
        return np.float32(0.0), int(cand.sum())

    def kept(lam):  # the product test in fp32: s2 >= fl(lam * ref)
        return int(np.sum(s2c >= np.float32(lam) * refc))

    lam = np.float32(ratios[target_count - 1])
    while kept(lam) < target_count:  # kept(0) counts every candidate (s2 >= 0)
        lam = np.nextafter(lam, np.float32(0.0))
    while True:                      # kept(+inf) is 0
        up = np.nextafter(lam, np.float32(np.inf))
        if kept(up) < target_count:
            break
        lam = up
    return np.float32(lam), int(cand.sum())


def mean_reference(s, unit_off, cand):
    """Mean-threshold reference (component ablation, "Mean threshold"): for
    each unit [unit_off[u], unit_off[u+1]) the mean of s over its candidate
    rows (``cand``: visual rows, restricted to S1 in Stage II); 0 for a unit
    without candidates. The threshold is then s(v) >= lambda * mean.
    """
    s = np.asarray(s, dtype=np.float64)
    cand = np.asarray(cand, dtype=bool)
    unit_off = as_i64(unit_off)
    ref = np.zeros(len(unit_off) - 1, dtype=np.float64)
    for u in range(len(unit_off) - 1):
        c = cand[unit_off[u]:unit_off[u + 1]]
        if c.any():
            ref[u] = np.mean(s[unit_off[u]:unit_off[u + 1]][c])
    return ref


def pool_scores(s, group: int, mode: str = "sum"):
    """Scores of merged tokens from the scores of their patches: rows
    [group i, group i + group) of ``s`` form merged row i, reduced by "sum"
    (the attention mass of the group), "mean" or "max". The row count must
    be a multiple of ``group``.
    """
    s = np.asarray(s, dtype=np.float64)
    assert group >= 1 and s.shape[0] % group == 0
    g = s.reshape(-1, group)
    if mode == "sum":
        return g.sum(axis=1)
    if mode == "mean":
        return g.mean(axis=1)
    if mode == "max":
        return g.max(axis=1)
    raise ValueError(mode)


def budget_keep(s, row_off, cand, budget, is_reg, keep_registers: bool = True):
    """Fixed-budget selection (Sec. 2, S = top-K(V, s); component ablation,
    "Fixed budget"): in sample b the min(budget[b], #candidates) candidate rows
    with the largest s. Candidates are ranked by score, high first, and equal
    scores by row id, low first; the first budget[b] of that order are kept.
    Register rows are kept iff ``keep_registers``. Returns (keep, count_vis).
    """
    s = np.asarray(s, dtype=np.float64)
    cand = np.asarray(cand, dtype=bool) & ~is_reg
    row_off = as_i64(row_off)
    keep = np.zeros(s.shape[0], dtype=bool)
    B = len(row_off) - 1
    count = np.zeros(B, dtype=np.int64)
    for b in range(B):
        rows = np.arange(row_off[b], row_off[b + 1])[cand[row_off[b]:row_off[b + 1]]]
        k = max(0, int(budget[b]))
        order = sorted(rows.tolist(), key=lambda r: (-s[r], r))
        chosen = order[:k]
        keep[chosen] = True
        count[b] = len(chosen)
    if keep_registers:
        keep |= is_reg
    return keep, count


# --------------------------------------------------------------------------- Stage II

def stage2_scores(Q_text, K_text, K2, keep1, is_reg, row_off, text_off,
                  text_keys: str = "causal", head_reduce: str = "mean"):
    """Stage-II text scores (Sec. 3.5, Eq. 7; App. A, Eqs. 15-16).

    For sample b the keys are the S1 rows (visual rows with keep1 and all
    registers, in row order) followed, for text token j, by the text keys
    0..j. Per head A = softmax(q_j k^T / sqrt(d2)); p[j, row] = mean_h A_h.
    K2 / K_text may hold fewer heads than Q_text (grouped-query attention);
    query head h then uses key head h // (H / H_kv).
    s2[v] = max_j p[j, v] for visual S1 rows (0 elsewhere) and
    ref2[b] = mean over the sample's registers of mean_j p[j, reg].
    Returns (s2 [rows], ref2 [B]).
    """
    Q = as_f64(Q_text)
    Kt = None if (K_text is None or text_keys == "none") else as_f64(K_text)
    K = as_f64(K2)
    row_off = as_i64(row_off)
    text_off = as_i64(text_off)
    keep1 = np.asarray(keep1, dtype=bool)
    B = row_off.shape[0] - 1
    # grouped-query attention: H query heads share H_kv key heads, query head h reading key head h // (H / H_kv)
    H, Hkv, d = Q.shape[1], K.shape[1], K.shape[2]
    assert H % Hkv == 0
    grp = H // Hkv
    scale = 1.0 / np.sqrt(d)
    s2 = np.zeros(K.shape[0], dtype=np.float64)
    ref2 = np.zeros(B, dtype=np.float64)
    for b in range(B):
        rows = np.arange(row_off[b], row_off[b + 1])
        in_s1 = (keep1[rows] & ~is_reg[rows]) | is_reg[rows]
        s1_rows = rows[in_s1]
        t0, t1 = text_off[b], text_off[b + 1]
        M = t1 - t0
        n = s1_rows.shape[0]
        p = np.zeros((M, n), dtype=np.float64)
        pmax = np.zeros((M, n), dtype=np.float64)
        for h in range(H):
            q = Q[t0:t1, h, :]                                # [M, d]
            li = (q @ K[s1_rows, h // grp, :].T) * scale      # [M, n]
            if Kt is not None:
                lt = (q @ Kt[t0:t1, h // grp, :].T) * scale   # [M, M]
                causal = np.tril(np.ones((M, M), dtype=bool))
                lt = np.where(causal, lt, -np.inf)
                A = softmax(np.concatenate([li, lt], axis=1), axis=1)[:, :n]
            else:
                A = softmax(li, axis=1)
            p += A / H
            pmax = np.maximum(pmax, A)
        vis = ~is_reg[s1_rows]
        if head_reduce == "mean":
            s2[s1_rows[vis]] = p[:, vis].max(axis=0) if M > 0 else 0.0
        elif head_reduce == "max":
            s2[s1_rows[vis]] = pmax[:, vis].max(axis=0) if M > 0 else 0.0
        else:
            raise ValueError(head_reduce)
        regs = ~vis
        ref2[b] = p[:, regs].mean(axis=0).mean() if M > 0 else 0.0
    return s2, ref2


# --------------------------------------------------------------------------- compaction

def compact(keep, row_off, tensors=()):
    """Order-preserving compaction of the kept rows (Algorithm 1: decode on [S2; T]).

    out_index lists the kept global row ids in ascending order (so sample-major);
    count_out[b] is the number of kept rows of sample b and out_off its prefix.
    Each tensor in ``tensors`` is gathered with the same index list (an exact
    copy of the rows).
    """
    keep = np.asarray(keep, dtype=bool)
    row_off = as_i64(row_off)
    B = row_off.shape[0] - 1
    out_index = np.nonzero(keep)[0].astype(np.int64)
    count_out = np.array([int(keep[row_off[b]:row_off[b + 1]].sum()) for b in range(B)], dtype=np.int64)
    out_off = np.concatenate([[0], np.cumsum(count_out)]).astype(np.int64)
    gathered = [np.asarray(t)[out_index] for t in tensors]
    return out_index, count_out, out_off, gathered


# --------------------------------------------------------------------------- full path

def near_threshold(s, tau, rel: float = 1e-5) -> np.ndarray:
    """Rows whose score lies within ``rel`` (relative) of their threshold."""
    s = np.asarray(s, dtype=np.float64)
    tau = np.asarray(tau, dtype=np.float64)
    return np.abs(s - tau) <= rel * np.abs(tau)


def prune(batch: dict, lambda1: float, lambda2: float, keep_registers: bool = True,
          text_keys: str = "causal", head_reduce: str = "mean", keep1_override=None,
          gather=("hidden", "K2", "V"), stage1: str | None = None, rule: str = "register",
          budget=None) -> dict:
    """Two-stage OccamToken pruning of one batch (Algorithm 1: Stage I, then Stage II).

    ``batch`` holds the synthetic tensors (any array type convertible to
    numpy) and its ``meta`` dict. ``keep1_override`` replaces the Stage-I
    decision (used to re-run Stage II on another Stage-I mask).
    ``rule``: "register" (the method, Eqs. 5 and 8), "mean" (both references
    replaced by mean_reference) or "budget" (Stage II replaced by
    budget_keep with the per-sample ``budget``).
    """
    meta = batch["meta"]
    rows = int(meta["total_rows"])
    seg_off = meta["seg_off_host"]
    row_off = meta["row_off_host"]
    reg_idx = meta["reg_idx_host"]
    reg_off = meta["reg_off_host"]
    text_off = meta["text_off_host"]
    is_reg = register_mask(rows, reg_idx)
    mode = stage1 or meta["stage1"]
    if mode == "cls":
        s1, ref1 = stage1_cls(batch["q_cls"], batch.get("k_cls"), batch["K1"], seg_off, reg_idx, reg_off)
    else:
        s1, ref1 = stage1_mutual(batch["Q1"], batch["K1"], seg_off, reg_idx, reg_off)
    seg_of_row = np.repeat(np.arange(len(seg_off) - 1), np.diff(seg_off))
    if rule == "mean":
        ref1 = mean_reference(s1, seg_off, ~is_reg)
    elif rule not in ("register", "budget"):
        raise ValueError(rule)
    tau1 = lambda1 * ref1[seg_of_row]
    # S1 = {v : s1(v) >= lambda1 s1(r)} u {r}: the registers are always in S1 (Eq. 5)
    keep1 = threshold(s1, ref1[seg_of_row], lambda1, is_reg, keep_registers=True)
    if keep1_override is not None:
        keep1 = (np.asarray(keep1_override, dtype=bool) & ~is_reg) | is_reg
    s2, ref2 = stage2_scores(batch["Q_text"], batch.get("K_text"), batch["K2"], keep1, is_reg,
                             row_off, text_off, text_keys=text_keys, head_reduce=head_reduce)
    sample_of_row = np.repeat(np.arange(len(row_off) - 1), np.diff(row_off))
    if rule == "mean":
        ref2 = mean_reference(s2, row_off, keep1 & ~is_reg)
    tau2 = lambda2 * ref2[sample_of_row]
    if rule == "budget":
        keep2, _ = budget_keep(s2, row_off, keep1, budget, is_reg, keep_registers=keep_registers)
    else:
        keep2 = threshold(s2, ref2[sample_of_row], lambda2, is_reg, prev_keep=keep1,
                          keep_registers=keep_registers)
    B = len(row_off) - 1
    count_vis = np.array([int((keep2 & ~is_reg)[row_off[b]:row_off[b + 1]].sum()) for b in range(B)])
    n1_vis = np.array([int((keep1 & ~is_reg)[row_off[b]:row_off[b + 1]].sum()) for b in range(B)])
    tensors = []
    names = []
    for g in gather:
        if g in batch:
            t = batch[g]
            if hasattr(t, "detach"):
                t = t.detach().cpu()
                t = t.view(t.shape[0], -1)
                import torch
                t = t.view(torch.int16).numpy()   # raw bit pattern: the copy is exact
            tensors.append(t)
            names.append(g)
    out_index, count_out, out_off, gathered = compact(keep2, row_off, tensors)
    near1 = near_threshold(s1, tau1) & ~is_reg
    near2 = near_threshold(s2, tau2) & keep1 & ~is_reg
    return dict(
        s1=s1, ref1=ref1, tau1=tau1, keep1=keep1,
        s2=s2, ref2=ref2, tau2=tau2, keep2=keep2, is_reg=is_reg,
        count_vis=count_vis, n1_vis=n1_vis, count_out=count_out, out_off=out_off,
        out_index=out_index, gathered=dict(zip(names, gathered)),
        near1=near1, near2=near2,
    )
