"""Seeded synthetic batches shaped like the paper's workloads.

Recipe (all random draws are seeded; shapes/counts use a numpy Generator so they
are identical on every machine, tensor values use a torch Generator on the
target device):

* every key/query/hidden/value element is i.i.d. N(0, 1) in fp32, rounded to
  bf16 (round-to-nearest-even) at the end;
* rows are laid out sample-major, segment-major: each segment (a crop or a
  frame) holds its P visual rows followed by its R register rows;
* sinks: chosen visual rows get their Stage-I key (K1) and Stage-II key (K2)
  vectors scaled by 8 (key norm x8);
* near-duplicates ("neighbour"): a chosen fraction of the rows at odd positions
  of a segment become rho * (previous row) + sqrt(1 - rho^2) * (own draw), in
  K1, K2, hidden and V alike, so the cosine to the neighbour is about rho;
* inter-frame duplicates ("frame"): the same construction against the row at
  the same position of the previous frame, applied frame after frame;
* registers: the register is the token that absorbs the sink-like attention
  mass (Sec. 2 "Test-time register token", App. A "Register construction").
  Its Stage-I key gets a component along the segment's [CLS] query (CLS mode)
  or along the segment's shared query component (mutual mode) sized so that
  the logit gains ``beta1``. Register Stage-II keys are plain N(0, 1);
* mutual mode: every query row of a segment carries a shared component of norm
  ``query_bias * sqrt(d1)`` along a random direction.

Nothing here computes attention, scores, thresholds or compaction.
"""

from __future__ import annotations

import math

import numpy as np
import torch

from .configs import Workload, get_config

BF16 = torch.bfloat16


def _shapes(w: Workload, rng: np.random.Generator):
    """Per-sample visual counts P_b (per segment) and text lengths M_b."""
    B = w.B
    if w.vis[0] == "fixed" and w.M[0] == "fixed" and w.vis[1] == 0:
        raise ValueError("explicit shapes required")
    if w.vis[0] == "fixed":
        P = np.full(B, w.vis[1], dtype=np.int64)
    elif w.vis[0] == "uniform_step":
        lo, hi, step = w.vis[1:]
        P = lo + step * rng.integers(0, (hi - lo) // step + 1, size=B)
    else:
        raise ValueError(w.vis)
    if w.M[0] == "fixed":
        M = np.full(B, w.M[1], dtype=np.int64)
    elif w.M[0] == "uniform":
        M = rng.integers(w.M[1], w.M[2] + 1, size=B)
    else:
        raise ValueError(w.M)
    return P.astype(np.int64), M.astype(np.int64)


def _layout(w: Workload, P: np.ndarray, M: np.ndarray):
    B, S_b, R = w.B, w.segs, w.regs
    seg_len = []
    seg_sample = []
    for b in range(B):
        for _ in range(S_b):
            seg_len.append(int(P[b]) + R)
            seg_sample.append(b)
    seg_len = np.asarray(seg_len, dtype=np.int64)
    seg_off = np.concatenate([[0], np.cumsum(seg_len)]).astype(np.int64)
    row_off = seg_off[:: S_b].copy()
    assert row_off.shape[0] == B + 1
    reg_idx = []
    for s in range(len(seg_len)):
        end = seg_off[s + 1]
        reg_idx.extend(range(int(end) - R, int(end)))
    reg_idx = np.asarray(reg_idx, dtype=np.int32)
    reg_off = (np.arange(len(seg_len) + 1) * R).astype(np.int32)
    text_off = np.concatenate([[0], np.cumsum(M)]).astype(np.int64)
    return dict(
        seg_off=seg_off, row_off=row_off, seg_sample=np.asarray(seg_sample, np.int32),
        reg_idx=reg_idx, reg_off=reg_off, text_off=text_off,
    )


def _choose_sinks(w: Workload, P: np.ndarray, lay: dict, rng: np.random.Generator) -> np.ndarray:
    rows = []
    for s in range(len(lay["seg_sample"])):
        b = lay["seg_sample"][s]
        p = int(P[b])
        if w.sinks[0] == "count":
            n = min(int(w.sinks[1]), p)
        else:
            n = max(1, int(round(w.sinks[1] * p)))
        pos = rng.choice(p, size=n, replace=False)
        rows.extend((lay["seg_off"][s] + np.sort(pos)).tolist())
    return np.asarray(rows, dtype=np.int64)


def _choose_dups(w: Workload, P: np.ndarray, lay: dict, rng: np.random.Generator):
    """Returns a list of (dst_rows, src_rows) index arrays, applied in order."""
    if w.dup is None:
        return []
    kind, frac, _rho = w.dup
    steps = []
    if kind == "neighbour":
        dst = []
        for s in range(len(lay["seg_sample"])):
            p = int(P[lay["seg_sample"][s]])
            odd = np.arange(1, p, 2)
            n = min(len(odd), int(round(frac * p)))
            pos = np.sort(rng.choice(odd, size=n, replace=False))
            dst.extend((lay["seg_off"][s] + pos).tolist())
        dst = np.asarray(dst, dtype=np.int64)
        steps.append((dst, dst - 1))
    elif kind == "frame":
        S_b = w.segs
        for f in range(1, S_b):
            dst, src = [], []
            for b in range(w.B):
                p = int(P[b])
                s = b * S_b + f
                n = int(round(frac * p))
                pos = np.sort(rng.choice(p, size=n, replace=False))
                dst.extend((lay["seg_off"][s] + pos).tolist())
                src.extend((lay["seg_off"][s - 1] + pos).tolist())
            steps.append((np.asarray(dst, np.int64), np.asarray(src, np.int64)))
    else:
        raise ValueError(kind)
    return steps


def _randn(gen: torch.Generator, shape, device) -> torch.Tensor:
    return torch.randn(*shape, generator=gen, device=device, dtype=torch.float32)


def _apply_dups(x: torch.Tensor, steps, rho: float) -> torch.Tensor:
    s = math.sqrt(1.0 - rho * rho)
    for dst, src in steps:
        d = torch.as_tensor(dst, device=x.device)
        sr = torch.as_tensor(src, device=x.device)
        x[d] = rho * x[sr] + s * x[d]
    return x


def _stage2(out, gen, T, rows, H2, H2kv, d2, device, dups, rho, sink_rows):
    out["Q_text"] = _randn(gen, (T, H2, d2), device).to(BF16)
    out["K_text"] = _randn(gen, (T, H2kv, d2), device).to(BF16)
    K2 = _randn(gen, (rows, H2kv, d2), device)
    K2 = _apply_dups(K2, dups, rho)
    K2[sink_rows] *= 8.0
    out["K2"] = K2.to(BF16)


def make_batch(w: Workload | str, device: str | torch.device = "cpu", seed: int | None = None,
               with_gather: bool = True, P=None, M=None, with_stage2: bool = True) -> dict:
    """Draw one synthetic batch for workload ``w`` on ``device``.

    Returns a dict of tensors (bf16 values, int offsets) plus a ``meta`` dict
    holding host copies of every offset array and the scalar sizes. ``P`` and
    ``M`` optionally fix the per-sample visual counts and text lengths.
    """
    if isinstance(w, str):
        w = get_config(w)
    seed = w.seed if seed is None else seed
    device = torch.device(device)
    rng = np.random.default_rng(seed)
    P0, M0 = _shapes(w, rng) if (P is None or M is None) else (None, None)
    P = P0 if P is None else np.asarray(P, np.int64)
    M = M0 if M is None else np.asarray(M, np.int64)
    lay = _layout(w, P, M)
    sinks = _choose_sinks(w, P, lay, rng)
    dups = _choose_dups(w, P, lay, rng)
    rho = w.dup[2] if w.dup else 0.0

    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) * 1000003 + 17)

    S_tot = len(lay["seg_sample"])
    rows = int(lay["seg_off"][-1])
    T = int(lay["text_off"][-1])
    H1, d1, H2, d2 = w.H1, w.d1, w.H2, w.d2
    reg_rows = torch.as_tensor(lay["reg_idx"].astype(np.int64), device=device)
    reg_seg = torch.as_tensor(np.repeat(np.arange(S_tot), w.regs), device=device)
    sink_rows = torch.as_tensor(sinks, device=device)

    out = {}
    # ---- Stage-I inputs
    K1 = _randn(gen, (rows, H1, d1), device)
    if w.stage1 == "cls":
        q_cls = _randn(gen, (S_tot, H1, d1), device)
        k_cls = _randn(gen, (S_tot, H1, d1), device)
        anchor = q_cls                                     # [S, H1, d1]
    else:
        Q1 = _randn(gen, (rows, H1, d1), device)
        direction = _randn(gen, (S_tot, H1, d1), device)
        direction = direction / direction.norm(dim=-1, keepdim=True)
        mu = w.query_bias * math.sqrt(d1) * direction     # [S, H1, d1]
        seg_of_row = torch.repeat_interleave(
            torch.arange(S_tot, device=device),
            torch.as_tensor(np.diff(lay["seg_off"]), device=device))
        Q1 += mu[seg_of_row]
        anchor = mu
    K1 = _apply_dups(K1, dups, rho)
    K1[sink_rows] *= 8.0
    a = anchor[reg_seg]                                    # [S*R, H1, d1]
    boost = w.beta1 * math.sqrt(d1) * a / (a * a).sum(-1, keepdim=True)
    K1[reg_rows] += boost
    out["K1"] = K1.to(BF16)
    del K1
    if w.stage1 == "cls":
        out["q_cls"] = q_cls.to(BF16)
        out["k_cls"] = k_cls.to(BF16)
    else:
        out["Q1"] = Q1.to(BF16)
        del Q1

    # ---- Stage-II inputs (layer-l queries/keys of the LLM)
    if not with_stage2:
        with_gather = False
    else:
        _stage2(out, gen, T, rows, H2, w.H2kv or H2, d2, device, dups, rho, sink_rows)

    # ---- rows gathered after pruning (hidden states and values of layer l)
    if with_gather:
        for name in ("hidden", "V"):
            x = _randn(gen, (rows, w.hidden), device)
            x = _apply_dups(x, dups, rho)
            out[name] = x.to(BF16)
            del x

    for k in ("row_off", "seg_off", "seg_sample", "reg_idx", "reg_off", "text_off"):
        out[k] = torch.as_tensor(lay[k], device=device)
    meta = dict(
        name=w.name, B=w.B, S_tot=S_tot, total_rows=rows, total_text=T,
        max_seg_rows=int(np.diff(lay["seg_off"]).max()),
        max_sample_rows=int(np.diff(lay["row_off"]).max()),
        max_text=int(M.max()), min_text=int(M.min()),
        regs_per_seg=w.regs, segs_per_sample=w.segs,
        H1=H1, d1=d1, H2=H2, d2=d2, H2kv=w.H2kv or H2, hidden=w.hidden, stage1=w.stage1,
        lambda1=w.lambda1, lambda2=w.lambda2, beta1=w.beta1,
        P=P, M=M, sinks=sinks, seed=seed,
        **{k + "_host": lay[k] for k in lay},
    )
    out["meta"] = meta
    return out


def tiny_batch(B=2, segs=2, P=(5, 7), R=2, M=(3, 4), H1=2, d1=8, H2=2, d2=8, hidden=16, H2kv=0,
               stage1="cls", seed=0, beta1=1.5, query_bias=0.5, sinks=("count", 1),
               dup=None, lambda1=0.5, lambda2=1.0) -> dict:
    """A small batch with explicit sizes (for oracle pins and ragged parity cases).

    ``P`` and ``M`` give per-sample visual counts (per segment) and text lengths.
    """
    P = tuple(P) if hasattr(P, "__len__") else (P,) * B
    M = tuple(M) if hasattr(M, "__len__") else (M,) * B
    assert len(P) == B and len(M) == B
    w = Workload(
        name="tiny", description="explicit small sizes", B=B, segs=segs, vis=("fixed", 0),
        regs=R, stage1=stage1, H1=H1, d1=d1, sinks=sinks, dup=dup, M=("fixed", 0), seed=seed,
        H2=H2, d2=d2, H2kv=H2kv, hidden=hidden, query_bias=query_bias, beta1=beta1,
        lambda1=lambda1, lambda2=lambda2,
    )
    return make_batch(w, "cpu", P=P, M=M)


def batch_slice_to_host(batch: dict, samples) -> dict:
    """Copy the rows of the chosen samples of ``batch`` to host memory.

    Offsets are re-based so the result is a self-contained batch; ``row_base``
    maps each kept sample back to its first row in the original batch.
    """
    meta = batch["meta"]
    samples = [int(s) for s in samples]
    S_b = meta["segs_per_sample"]
    R = meta["regs_per_seg"]
    row_off = meta["row_off_host"]
    text_off = meta["text_off_host"]
    seg_off = meta["seg_off_host"]
    out = {}
    rows_sel, text_sel, segs_sel = [], [], []
    for b in samples:
        rows_sel.append(np.arange(row_off[b], row_off[b + 1]))
        text_sel.append(np.arange(text_off[b], text_off[b + 1]))
        segs_sel.append(np.arange(b * S_b, (b + 1) * S_b))
    rows_sel = np.concatenate(rows_sel)
    text_sel = np.concatenate(text_sel)
    segs_sel = np.concatenate(segs_sel)
    ri = torch.as_tensor(rows_sel, device=batch["K1"].device)
    ti = torch.as_tensor(text_sel, device=batch["K1"].device)
    si = torch.as_tensor(segs_sel, device=batch["K1"].device)
    for k in ("K1", "K2", "Q1", "hidden", "V"):
        if k in batch:
            out[k] = batch[k].index_select(0, ri).cpu()
    for k in ("q_cls", "k_cls"):
        if k in batch:
            out[k] = batch[k].index_select(0, si).cpu()
    for k in ("Q_text", "K_text"):
        out[k] = batch[k].index_select(0, ti).cpu()
    seg_len = np.diff(seg_off)[segs_sel]
    n_rows = np.diff(row_off)[samples]
    n_text = np.diff(text_off)[samples]
    new_seg_off = np.concatenate([[0], np.cumsum(seg_len)]).astype(np.int64)
    new_row_off = np.concatenate([[0], np.cumsum(n_rows)]).astype(np.int64)
    new_text_off = np.concatenate([[0], np.cumsum(n_text)]).astype(np.int64)
    reg_idx = []
    for s in range(len(segs_sel)):
        reg_idx.extend(range(int(new_seg_off[s + 1]) - R, int(new_seg_off[s + 1])))
    lay = dict(
        row_off=new_row_off, seg_off=new_seg_off,
        seg_sample=np.repeat(np.arange(len(samples)), S_b).astype(np.int32),
        reg_idx=np.asarray(reg_idx, np.int32),
        reg_off=(np.arange(len(segs_sel) + 1) * R).astype(np.int32),
        text_off=new_text_off,
    )
    for k, v in lay.items():
        out[k] = torch.as_tensor(v)
    m = dict(meta)
    m.update(
        B=len(samples), S_tot=len(segs_sel), total_rows=int(new_row_off[-1]),
        total_text=int(new_text_off[-1]), max_seg_rows=int(seg_len.max()),
        max_sample_rows=int(n_rows.max()), max_text=int(n_text.max()), min_text=int(n_text.min()),
        P=np.asarray(meta["P"])[samples], M=np.asarray(meta["M"])[samples],
        row_base=np.asarray(row_off)[samples],
        **{k + "_host": v for k, v in lay.items()},
    )
    out["meta"] = m
    return out
