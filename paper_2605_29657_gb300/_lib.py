"""ctypes binding of liboccam.so (include/occam.h).

Argument marshalling only: every step of the prune path runs in the CUDA
kernels behind the C ABI. PyTorch supplies device memory and the current
stream. There is no CPU fallback: if the library is missing or no CUDA device
is present, every call raises OccamError.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liboccam.so")

OCCAM_OK = 0
OCCAM_ERR_INVALID_ARG = 1
OCCAM_ERR_CAPACITY = 2
OCCAM_ERR_CUDA = 3
OCCAM_ERR_TIMEOUT = 4
OCCAM_ERR_UNSUPPORTED = 5
OCCAM_ERR_WORKSPACE = 6
ERROR_NAMES = {
    0: "OK", 1: "INVALID_ARG", 2: "CAPACITY", 3: "CUDA", 4: "TIMEOUT", 5: "UNSUPPORTED", 6: "WORKSPACE",
}
OCCAM_STAGE1_CLS = 0
OCCAM_STAGE1_MUTUAL = 1
OCCAM_REF_SEGMENT = 0
OCCAM_REF_SAMPLE = 1
OCCAM_ROUTE_AUTO, OCCAM_ROUTE_TWOPASS, OCCAM_ROUTE_NARROW = 0, 1, 2
OCCAM_MAX_GATHER = 8
OCCAM_RULE_REGISTER = 0
OCCAM_RULE_MEAN = 1
OCCAM_RULE_BUDGET = 2
RULES = {"register": OCCAM_RULE_REGISTER, "mean": OCCAM_RULE_MEAN, "budget": OCCAM_RULE_BUDGET}
POOLS = {"sum": 0, "mean": 1, "max": 2}

_p = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64


class OccamError(RuntimeError):
    def __init__(self, code: int, where: str = ""):
        self.code = code
        super().__init__(f"{where}: {ERROR_NAMES.get(code, code)} ({code})")


class CBatch(ctypes.Structure):
    _fields_ = [
        ("B", _i32), ("S_tot", _i32), ("total_rows", _i64), ("total_text", _i64),
        ("max_seg_rows", _i32), ("max_sample_rows", _i32), ("max_text", _i32), ("max_regs", _i32),
        ("row_off", _p), ("seg_off", _p), ("seg_first", _p), ("seg_sample", _p),
        ("reg_idx", _p), ("reg_off", _p), ("text_off", _p),
    ]


class CStage1(ctypes.Structure):
    _fields_ = [("mode", _i32), ("H1", _i32), ("d1", _i32), ("q", _p), ("k_cls", _p), ("K1", _p)]


class CStage2(ctypes.Structure):
    _fields_ = [("H2", _i32), ("d2", _i32), ("Q_text", _p), ("K_text", _p), ("K2", _p), ("H2_kv", _i32)]


class CPruneArgs(ctypes.Structure):
    _fields_ = [
        ("batch", CBatch), ("stage1", CStage1), ("stage2", CStage2),
        ("lambda1", ctypes.c_float), ("lambda2", ctypes.c_float),
        ("keep_registers", _i32), ("n_tensors", _i32),
        ("src", _p * OCCAM_MAX_GATHER), ("row_bytes", _i64 * OCCAM_MAX_GATHER), ("dst", _p * OCCAM_MAX_GATHER),
        ("capacity_rows", _i64), ("rule", _i32), ("budget", _p), ("near_rel", ctypes.c_float),
    ]


class CPruneOut(ctypes.Structure):
    _fields_ = [
        ("keep2", _p), ("out_index", _p), ("count_vis", _p), ("count_out", _p), ("out_off", _p),
        ("keep1", _p), ("s1", _p), ("ref1", _p), ("s2", _p), ("ref2", _p), ("n1_vis", _p), ("n_eff", _p),
        ("near1", _p), ("near2", _p),
    ]


_lib = None


def use_library(path: str) -> None:
    """Selects the shared library the binding loads (for example the
    bounds-checked build, liboccam_checked.so). Must come before the first
    call into the library."""
    global LIB_PATH
    if _lib is not None and os.path.abspath(path) != os.path.abspath(LIB_PATH):
        raise OccamError(OCCAM_ERR_INVALID_ARG, f"the library is already loaded from {LIB_PATH}")
    LIB_PATH = path


def library() -> ctypes.CDLL:
    """Loads liboccam.so once; raises OccamError when it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise OccamError(OCCAM_ERR_UNSUPPORTED,
                             f"liboccam.so not found at {LIB_PATH}; build it with paper_2605_29657_gb300.build.build()")
        lib = ctypes.CDLL(LIB_PATH)
        P = ctypes.POINTER
        lib.occam_version.restype = ctypes.c_char_p
        lib.occam_workspace_size.argtypes = [P(CBatch), _i32, _i32, P(ctypes.c_size_t)]
        lib.occam_get_status.argtypes = [_p, P(_i32), _p]
        lib.occam_score_stage1.argtypes = [P(CBatch), P(CStage1), _p, _p, _p, ctypes.c_size_t, _p]
        lib.occam_threshold.argtypes = [P(CBatch), _p, _p, _i32, ctypes.c_float, _p, _i32, _p, _p, _p,
                                        ctypes.c_size_t, _p]
        lib.occam_score_stage2.argtypes = [P(CBatch), P(CStage2), _p, _p, _p, _p, ctypes.c_size_t, _p]
        lib.occam_compact.argtypes = [P(CBatch), _p, _i32, P(_p), P(_i64), P(_p), _i64, _p, _p, _p, _p,
                                      ctypes.c_size_t, _p]
        lib.occam_prune.argtypes = [P(CPruneArgs), P(CPruneOut), _p, ctypes.c_size_t, _p]
        lib.occam_compact_noalloc.argtypes = [P(CBatch), _p, _i32, P(_p), P(_i64), P(_p), _i64, _p, _p, _p, _p]
        lib.occam_prune_traced.argtypes = [P(CPruneArgs), P(CPruneOut), _p, ctypes.c_size_t, _p, P(_p), _i32]
        lib.occam_prune_staged.argtypes = [P(CPruneArgs), P(CPruneOut), _p, ctypes.c_size_t, _p, ctypes.c_size_t,
                                           _p]
        lib.occam_calibrate_lambda2.argtypes = [P(CBatch), _p, _p, _p, _i64, _p, _p, _p, ctypes.c_size_t, _p]
        lib.occam_construct_registers.argtypes = [P(CBatch), _p, _i64, _p, _i32, _p, ctypes.c_size_t, _p]
        lib.occam_mean_reference.argtypes = [P(CBatch), _p, _i32, _p, _p, _p, ctypes.c_size_t, _p]
        lib.occam_budget_keep.argtypes = [P(CBatch), _p, _p, _p, _i32, _p, _p, _p, ctypes.c_size_t, _p]
        lib.occam_pool_scores.argtypes = [_p, _i64, _i32, _i32, _p, _p]
        lib.occam_selftest_wait.argtypes = [ctypes.c_uint64, _p, _p]
        lib.occam_last_call_kernels.argtypes = []
        lib.occam_set_stage2_route.argtypes = [_i32, P(_i32)]
        for name in ("occam_last_call_kernels", "occam_selftest_wait", "occam_pool_scores", "occam_mean_reference", "occam_budget_keep", "occam_construct_registers", "occam_calibrate_lambda2", "occam_workspace_size", "occam_get_status", "occam_score_stage1",
                     "occam_threshold",
                     "occam_score_stage2", "occam_compact", "occam_prune", "occam_prune_traced",
                     "occam_compact_noalloc", "occam_prune_staged", "occam_set_stage2_route"):
            getattr(lib, name).restype = ctypes.c_int
        _lib = lib
    return _lib


def _check(rc: int, where: str):
    if rc != OCCAM_OK:
        raise OccamError(rc, where)


def _ptr(t) -> int | None:
    if t is None:
        return None
    return t.data_ptr()


def _dev_tensor(t: torch.Tensor, dtype, name: str) -> torch.Tensor:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise OccamError(OCCAM_ERR_INVALID_ARG, f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise OccamError(OCCAM_ERR_INVALID_ARG, f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise OccamError(OCCAM_ERR_INVALID_ARG, f"{name} must be contiguous")
    return t


def _host_or_dev_tensor(t: torch.Tensor, dtype, name: str) -> torch.Tensor:
    """A CUDA tensor, or a pinned host tensor the device can read in place."""
    if isinstance(t, torch.Tensor) and not t.is_cuda:
        if not t.is_pinned():
            raise OccamError(OCCAM_ERR_INVALID_ARG, f"{name} must be a CUDA tensor or pinned host memory")
        if t.dtype != dtype or not t.is_contiguous():
            raise OccamError(OCCAM_ERR_INVALID_ARG, f"{name} must be contiguous {dtype}")
        return t
    return _dev_tensor(t, dtype, name)


def _stream(stream) -> int | None:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


class BatchLayout:
    """Device copy of a batch's row / segment / register / text layout.

    ``row_off`` [B+1], ``seg_off`` [S+1], ``reg_idx``, ``reg_off`` [S+1] and
    ``text_off`` [B+1] are host arrays; segments of one sample must be
    consecutive and tile the sample's rows.
    """

    def __init__(self, row_off, seg_off, reg_idx, reg_off, text_off, device="cuda"):
        row_off = np.asarray(row_off, np.int64)
        seg_off = np.asarray(seg_off, np.int64)
        reg_idx = np.asarray(reg_idx, np.int32)
        reg_off = np.asarray(reg_off, np.int32)
        text_off = np.asarray(text_off, np.int64)
        B = row_off.shape[0] - 1
        S = seg_off.shape[0] - 1
        if B < 1 or S < B or reg_off.shape[0] != S + 1:
            raise OccamError(OCCAM_ERR_INVALID_ARG, "layout sizes")
        seg_first = np.searchsorted(seg_off, row_off).astype(np.int32)
        if not np.array_equal(seg_off[seg_first], row_off):
            raise OccamError(OCCAM_ERR_INVALID_ARG, "segments must tile the samples")
        seg_sample = (np.searchsorted(row_off, seg_off[:-1], side="right") - 1).astype(np.int32)
        seg_len = np.diff(seg_off)
        n_text = np.diff(text_off)
        regs = np.diff(reg_off)
        if (seg_len < 1).any() or (regs < 1).any() or (n_text < 1).any():
            raise OccamError(OCCAM_ERR_INVALID_ARG, "every segment needs >= 1 row and >= 1 register; every sample >= 1 text token")
        self.B, self.S_tot = B, S
        self.total_rows = int(row_off[-1])
        self.total_text = int(text_off[-1])
        self.max_seg_rows = int(seg_len.max())
        self.max_sample_rows = int(np.diff(row_off).max())
        self.max_text = int(n_text.max())
        self.max_regs = int(regs.max())
        self.host = dict(row_off=row_off, seg_off=seg_off, seg_first=seg_first, seg_sample=seg_sample,
                         reg_idx=reg_idx, reg_off=reg_off, text_off=text_off)
        self.dev = {k: torch.as_tensor(v).to(device) for k, v in self.host.items()}
        self.device = torch.device(device)

    @classmethod
    def from_batch(cls, batch: dict, device="cuda") -> "BatchLayout":
        m = batch["meta"]
        return cls(m["row_off_host"], m["seg_off_host"], m["reg_idx_host"], m["reg_off_host"],
                   m["text_off_host"], device=device)

    def c(self) -> CBatch:
        d = self.dev
        return CBatch(self.B, self.S_tot, self.total_rows, self.total_text, self.max_seg_rows,
                      self.max_sample_rows, self.max_text, self.max_regs,
                      _ptr(d["row_off"]), _ptr(d["seg_off"]), _ptr(d["seg_first"]), _ptr(d["seg_sample"]),
                      _ptr(d["reg_idx"]), _ptr(d["reg_off"]), _ptr(d["text_off"]))


# ------------------------------------------------------------------ entry points (same names as the C ABI)

def occam_version() -> str:
    return library().occam_version().decode()


def occam_workspace_size(layout: BatchLayout, H1: int, H2: int) -> int:
    n = ctypes.c_size_t(0)
    cb = layout.c()
    _check(library().occam_workspace_size(ctypes.byref(cb), H1, H2, ctypes.byref(n)), "occam_workspace_size")
    return int(n.value)


def alloc_workspace(layout: BatchLayout, H1: int = 16, H2: int = 32) -> torch.Tensor:
    """A zero-filled, 256-byte aligned workspace (zero-filled before its first use, as the ABI requires)."""
    n = occam_workspace_size(layout, H1, H2)
    ws = torch.zeros(n + 256, dtype=torch.uint8, device=layout.device)
    off = (-ws.data_ptr()) % 256
    return ws[off:off + n]


def occam_get_status(ws: torch.Tensor, stream=None) -> int:
    v = _i32(0)
    _check(library().occam_get_status(_ptr(ws), ctypes.byref(v), _stream(stream)), "occam_get_status")
    return int(v.value)


def _ws(ws, layout, H1, H2):
    return alloc_workspace(layout, H1, H2) if ws is None else ws


def occam_score_stage1(layout: BatchLayout, mode: int, q, K1, k_cls=None, s1=None, ref1=None, ws=None,
                       stream=None):
    bf = torch.bfloat16
    _dev_tensor(q, bf, "q"); _dev_tensor(K1, bf, "K1")
    if k_cls is not None:
        _dev_tensor(k_cls, bf, "k_cls")
    H1, d1 = int(K1.shape[1]), int(K1.shape[2])
    dev = layout.device
    s1 = torch.empty(layout.total_rows, dtype=torch.float32, device=dev) if s1 is None else s1
    ref1 = torch.empty(layout.S_tot, dtype=torch.float32, device=dev) if ref1 is None else ref1
    ws = _ws(ws, layout, H1, 1)
    cb = layout.c()
    a = CStage1(mode, H1, d1, _ptr(q), _ptr(k_cls), _ptr(K1))
    _check(library().occam_score_stage1(ctypes.byref(cb), ctypes.byref(a), _ptr(s1), _ptr(ref1), _ptr(ws),
                                        ws.numel(), _stream(stream)), "occam_score_stage1")
    return s1, ref1


def occam_threshold(layout: BatchLayout, s, ref, ref_scope: int, lam: float, prev_keep=None,
                    keep_registers: bool = True, keep=None, count_vis=None, ws=None, stream=None):
    _dev_tensor(s, torch.float32, "s"); _dev_tensor(ref, torch.float32, "ref")
    dev = layout.device
    keep = torch.empty(layout.total_rows, dtype=torch.uint8, device=dev) if keep is None else keep
    count_vis = torch.empty(layout.B, dtype=torch.int32, device=dev) if count_vis is None else count_vis
    ws = _ws(ws, layout, 1, 1)
    cb = layout.c()
    _check(library().occam_threshold(ctypes.byref(cb), _ptr(s), _ptr(ref), int(ref_scope), float(lam),
                                     _ptr(prev_keep), int(bool(keep_registers)), _ptr(keep), _ptr(count_vis),
                                     _ptr(ws), ws.numel(), _stream(stream)), "occam_threshold")
    return keep, count_vis


def occam_mean_reference(layout: BatchLayout, s, ref_scope: int, prev_keep=None, ref=None, ws=None, stream=None):
    """Mean-threshold reference: per segment (OCCAM_REF_SEGMENT) or sample
    (OCCAM_REF_SAMPLE) the mean of s over the visual rows with prev_keep."""
    _dev_tensor(s, torch.float32, "s")
    if prev_keep is not None:
        _dev_tensor(prev_keep, torch.uint8, "prev_keep")
    n = layout.S_tot if ref_scope == OCCAM_REF_SEGMENT else layout.B
    ref = torch.empty(n, dtype=torch.float32, device=layout.device) if ref is None else ref
    ws = _ws(ws, layout, 1, 1)
    cb = layout.c()
    _check(library().occam_mean_reference(ctypes.byref(cb), _ptr(s), int(ref_scope), _ptr(prev_keep), _ptr(ref),
                                          _ptr(ws), ws.numel(), _stream(stream)), "occam_mean_reference")
    return ref


def occam_last_call_kernels() -> int:
    """Kernels the last entry point called on this thread launched."""
    return int(library().occam_last_call_kernels())


def occam_set_stage2_route(route: int) -> int:
    """Stage-II routing for tests and diagnostics (OCCAM_ROUTE_AUTO is the
    default). Returns the route in force before the call."""
    prev = _i32(0)
    _check(library().occam_set_stage2_route(int(route), ctypes.byref(prev)), "occam_set_stage2_route")
    return int(prev.value)


def occam_selftest_wait(limit_ns: int = 20_000_000, device="cuda", stream=None) -> tuple[int, int]:
    """Runs the bounded-wait diagnostic; returns (mask of the waits that gave
    up, status): (7, OCCAM_ERR_TIMEOUT) when every wait ran out as designed."""
    scratch = torch.empty(4, dtype=torch.int32, device=device)
    _check(library().occam_selftest_wait(int(limit_ns), _ptr(scratch), _stream(stream)), "occam_selftest_wait")
    out = scratch.cpu()
    return int(out[0]), int(out[1])


def occam_pool_scores(s, group: int, mode: str = "sum", out=None, stream=None) -> torch.Tensor:
    """Merged-token scores: the sum (default), mean or max of every group of
    `group` consecutive rows of s (a 2x2 patch merger's four patches)."""
    _dev_tensor(s, torch.float32, "s")
    if mode not in POOLS:
        raise OccamError(OCCAM_ERR_INVALID_ARG, f"mode must be one of {sorted(POOLS)}")
    if group < 1 or s.numel() % group:
        raise OccamError(OCCAM_ERR_INVALID_ARG, "the row count must be a multiple of group")
    out = torch.empty(s.numel() // group, dtype=torch.float32, device=s.device) if out is None else out
    _check(library().occam_pool_scores(_ptr(s), s.numel(), int(group), POOLS[mode], _ptr(out), _stream(stream)),
           "occam_pool_scores")
    return out


def occam_budget_keep(layout: BatchLayout, s, budget, prev_keep=None, keep_registers: bool = True, keep=None,
                      count_vis=None, ws=None, stream=None):
    """Fixed-budget rule: per sample the budget[b] candidates (visual rows with
    prev_keep) with the largest s, equal scores lower row first."""
    _dev_tensor(s, torch.float32, "s")
    _dev_tensor(budget, torch.int32, "budget")
    if prev_keep is not None:
        _dev_tensor(prev_keep, torch.uint8, "prev_keep")
    if budget.numel() != layout.B:
        raise OccamError(OCCAM_ERR_INVALID_ARG, "budget must have one entry per sample")
    dev = layout.device
    keep = torch.empty(layout.total_rows, dtype=torch.uint8, device=dev) if keep is None else keep
    count_vis = torch.empty(layout.B, dtype=torch.int32, device=dev) if count_vis is None else count_vis
    ws = _ws(ws, layout, 1, 1)
    cb = layout.c()
    _check(library().occam_budget_keep(ctypes.byref(cb), _ptr(s), _ptr(prev_keep), _ptr(budget),
                                       int(bool(keep_registers)), _ptr(keep), _ptr(count_vis), _ptr(ws),
                                       ws.numel(), _stream(stream)), "occam_budget_keep")
    return keep, count_vis


def occam_score_stage2(layout: BatchLayout, Q_text, K2, keep1, K_text=None, s2=None, ref2=None, ws=None,
                       stream=None):
    bf = torch.bfloat16
    _dev_tensor(Q_text, bf, "Q_text"); _dev_tensor(K2, bf, "K2"); _dev_tensor(keep1, torch.uint8, "keep1")
    if K_text is not None:
        _dev_tensor(K_text, bf, "K_text")
    # query heads from Q_text, key heads from K2 (fewer under grouped-query attention)
    H2, d2, H2kv = int(Q_text.shape[1]), int(K2.shape[2]), int(K2.shape[1])
    dev = layout.device
    s2 = torch.empty(layout.total_rows, dtype=torch.float32, device=dev) if s2 is None else s2
    ref2 = torch.empty(layout.B, dtype=torch.float32, device=dev) if ref2 is None else ref2
    ws = _ws(ws, layout, 1, H2)
    cb = layout.c()
    a = CStage2(H2, d2, _ptr(Q_text), _ptr(K_text), _ptr(K2), H2kv)
    _check(library().occam_score_stage2(ctypes.byref(cb), ctypes.byref(a), _ptr(keep1), _ptr(s2), _ptr(ref2),
                                        _ptr(ws), ws.numel(), _stream(stream)), "occam_score_stage2")
    return s2, ref2


def occam_construct_registers(layout: BatchLayout, h, k_reg, ws=None, stream=None) -> torch.Tensor:
    """Test-time register construction in place on h [total_rows, channels]
    bf16 (Algorithm 1, step 2): per segment and channel in k_reg, the
    registers take the visual rows' max, which is then zeroed on them."""
    h = _dev_tensor(h, torch.bfloat16, "h")
    k_reg = _dev_tensor(k_reg, torch.int32, "k_reg")
    if h.dim() != 2 or h.shape[0] != layout.total_rows:
        raise OccamError(OCCAM_ERR_INVALID_ARG, "h must be [total_rows, channels]")
    if k_reg.numel() and (int(k_reg.min()) < 0 or int(k_reg.max()) >= h.shape[1]):
        raise OccamError(OCCAM_ERR_INVALID_ARG, "k_reg channels out of range")
    if k_reg.numel() != torch.unique(k_reg).numel():
        raise OccamError(OCCAM_ERR_INVALID_ARG, "k_reg channels must be distinct")
    ws = _ws(ws, layout, 1, 1)
    cb = layout.c()
    _check(library().occam_construct_registers(ctypes.byref(cb), _ptr(h), int(h.shape[1]), _ptr(k_reg),
                                               int(k_reg.numel()), _ptr(ws), ws.numel(), _stream(stream)),
           "occam_construct_registers")
    return h


def occam_calibrate_lambda2(layout: BatchLayout, s2, ref2, keep1, target_count: int, ws=None,
                            stream=None) -> tuple[torch.Tensor, torch.Tensor]:
    """lambda2 matching a total retained budget over the batch (App. A): the
    target_count-th largest s2 / ref2 ratio of the visual S1 rows. Returns
    (lambda2 [1] fp32, candidate count [1] int32), both on the device."""
    s2 = _dev_tensor(s2, torch.float32, "s2")
    ref2 = _dev_tensor(ref2, torch.float32, "ref2")
    keep1 = _dev_tensor(keep1, torch.uint8, "keep1")
    ws = _ws(ws, layout, 1, 1)
    lam = torch.empty(1, dtype=torch.float32, device=layout.device)
    n = torch.empty(1, dtype=torch.int32, device=layout.device)
    cb = layout.c()
    _check(library().occam_calibrate_lambda2(ctypes.byref(cb), _ptr(s2), _ptr(ref2), _ptr(keep1),
                                             int(target_count), _ptr(lam), _ptr(n), _ptr(ws), ws.numel(),
                                             _stream(stream)), "occam_calibrate_lambda2")
    return lam, n


def _gather_arrays(tensors, dsts):
    n = len(tensors)
    if n > OCCAM_MAX_GATHER:
        raise OccamError(OCCAM_ERR_INVALID_ARG, "too many gather tensors")
    src = (_p * max(n, 1))(*[_ptr(t) for t in tensors])
    dst = (_p * max(n, 1))(*[_ptr(t) for t in dsts])
    rb = (_i64 * max(n, 1))(*[t.stride(0) * t.element_size() for t in tensors])
    return n, src, rb, dst


def occam_compact(layout: BatchLayout, keep, tensors=(), capacity_rows: int | None = None, dst=None,
                  out_index=None, count_out=None, out_off=None, ws=None, stream=None):
    _dev_tensor(keep, torch.uint8, "keep")
    dev = layout.device
    cap = layout.total_rows if capacity_rows is None else int(capacity_rows)
    tensors = [_dev_tensor(t, t.dtype, f"tensor{i}") for i, t in enumerate(tensors)]
    if dst is None:
        dst = [torch.empty((cap,) + tuple(t.shape[1:]), dtype=t.dtype, device=dev) for t in tensors]
    out_index = torch.empty(max(cap, 1), dtype=torch.int32, device=dev) if out_index is None else out_index
    count_out = torch.empty(layout.B, dtype=torch.int32, device=dev) if count_out is None else count_out
    out_off = torch.empty(layout.B + 1, dtype=torch.int64, device=dev) if out_off is None else out_off
    ws = _ws(ws, layout, 1, 1)
    n, src_a, rb_a, dst_a = _gather_arrays(tensors, dst)
    cb = layout.c()
    _check(library().occam_compact(ctypes.byref(cb), _ptr(keep), n, src_a, rb_a, dst_a, cap, _ptr(out_index),
                                   _ptr(count_out), _ptr(out_off), _ptr(ws), ws.numel(), _stream(stream)),
           "occam_compact")
    return dict(out_index=out_index, count_out=count_out, out_off=out_off, gathered=dst)


def occam_compact_noalloc(layout: BatchLayout, keep, tensors=(), capacity_rows: int | None = None, dst=None,
                          out_index=None, count_out=None, out_off=None, stream=None):
    """occam_compact without a workspace, for callers that cannot allocate
    device memory: the library's own fixed scratch array is used instead.
    Output buffers are the caller's; pass them in to allocate nothing here."""
    _dev_tensor(keep, torch.uint8, "keep")
    dev = layout.device
    cap = layout.total_rows if capacity_rows is None else int(capacity_rows)
    tensors = [_dev_tensor(t, t.dtype, f"tensor{i}") for i, t in enumerate(tensors)]
    if dst is None:
        dst = [torch.empty((cap,) + tuple(t.shape[1:]), dtype=t.dtype, device=dev) for t in tensors]
    out_index = torch.empty(max(cap, 1), dtype=torch.int32, device=dev) if out_index is None else out_index
    count_out = torch.empty(layout.B, dtype=torch.int32, device=dev) if count_out is None else count_out
    out_off = torch.empty(layout.B + 1, dtype=torch.int64, device=dev) if out_off is None else out_off
    n, src_a, rb_a, dst_a = _gather_arrays(tensors, dst)
    cb = layout.c()
    _check(library().occam_compact_noalloc(ctypes.byref(cb), _ptr(keep), n, src_a, rb_a, dst_a, cap,
                                           _ptr(out_index), _ptr(count_out), _ptr(out_off), _stream(stream)),
           "occam_compact_noalloc")
    return dict(out_index=out_index, count_out=count_out, out_off=out_off, gathered=dst)


class PruneCall:
    """A prepared occam_prune call: argument structs, outputs and workspace are
    built once and reused, so repeated calls marshal nothing."""

    OPTIONAL = ("keep1", "s1", "ref1", "s2", "ref2", "n1_vis", "n_eff")  # n_eff: [CLS] mode only
    NEAR = ("near1", "near2")  # near-threshold flags of the two tests (opt-in through `want`)

    def __init__(self, layout: BatchLayout, stage1: dict, stage2: dict, lambda1: float, lambda2: float,
                 keep_registers: bool = True, gather=(), capacity_rows: int | None = None,
                 want=OPTIONAL, ws=None, host_inputs: bool = False, rule: str = "register", budget=None,
                 near_rel: float = 0.0):
        """host_inputs: K2 and the gather tensors may be pinned host tensors,
        read in place through occam_prune_staged (S1 rows of K2 and kept rows
        only); a device staging tensor for K2 is allocated here.
        rule: "register" (the method), "mean" or "budget" (the component
        ablation's variants); budget: [B] int32 CUDA tensor for "budget".
        want may name "near1" / "near2" (PruneCall.NEAR): the near-threshold
        flags of the two tests, with relative band near_rel (0: 1e-5)."""
        bf = torch.bfloat16
        mode = OCCAM_STAGE1_CLS if stage1.get("mode", "cls") == "cls" else OCCAM_STAGE1_MUTUAL
        q = _dev_tensor(stage1["q"], bf, "q")
        K1 = _dev_tensor(stage1["K1"], bf, "K1")
        k_cls = stage1.get("k_cls")
        if k_cls is not None:
            _dev_tensor(k_cls, bf, "k_cls")
        Q_text = _dev_tensor(stage2["Q_text"], bf, "Q_text")
        K2 = (_host_or_dev_tensor if host_inputs else _dev_tensor)(stage2["K2"], bf, "K2")
        K_text = stage2.get("K_text")
        if K_text is not None:
            _dev_tensor(K_text, bf, "K_text")
        H1, d1 = int(K1.shape[1]), int(K1.shape[2])
        # query heads from Q_text, key heads from K2 (fewer under grouped-query attention)
        H2, d2, H2kv = int(Q_text.shape[1]), int(K2.shape[2]), int(K2.shape[1])
        dev = layout.device
        self.layout = layout
        self.keep_alive = [q, K1, k_cls, Q_text, K2, K_text]
        cap = layout.total_rows if capacity_rows is None else int(capacity_rows)
        check = _host_or_dev_tensor if host_inputs else _dev_tensor
        gather = [check(t, t.dtype, f"gather{i}") for i, t in enumerate(gather)]
        self.k2_stage = torch.empty(K2.shape, dtype=bf, device=dev) if host_inputs else None
        self.gathered = [torch.empty((cap,) + tuple(t.shape[1:]), dtype=t.dtype, device=dev) for t in gather]
        self.keep_alive += gather
        R, B = layout.total_rows, layout.B
        o = dict(
            keep2=torch.empty(R, dtype=torch.uint8, device=dev),
            out_index=torch.empty(max(cap, 1), dtype=torch.int32, device=dev),
            count_vis=torch.empty(B, dtype=torch.int32, device=dev),
            count_out=torch.empty(B, dtype=torch.int32, device=dev),
            out_off=torch.empty(B + 1, dtype=torch.int64, device=dev),
        )
        shapes = dict(keep1=(R, torch.uint8), s1=(R, torch.float32), ref1=(layout.S_tot, torch.float32),
                      s2=(R, torch.float32), ref2=(B, torch.float32), n1_vis=(B, torch.int32),
                      n_eff=((layout.S_tot, H1), torch.float32), near1=(R, torch.uint8), near2=(R, torch.uint8))
        if mode != OCCAM_STAGE1_CLS:
            want = tuple(k for k in want if k != "n_eff")
        for k in want:
            n, dt = shapes[k]
            o[k] = torch.empty(n, dtype=dt, device=dev)
        self.out = o
        self.ws = alloc_workspace(layout, H1, H2) if ws is None else ws
        n, src_a, rb_a, dst_a = _gather_arrays(gather, self.gathered)
        a = CPruneArgs()
        a.batch = layout.c()
        a.stage1 = CStage1(mode, H1, d1, _ptr(q), _ptr(k_cls), _ptr(K1))
        a.stage2 = CStage2(H2, d2, _ptr(Q_text), _ptr(K_text), _ptr(K2), H2kv)
        a.lambda1 = float(lambda1)
        a.lambda2 = float(lambda2)
        a.keep_registers = int(bool(keep_registers))
        a.n_tensors = n
        for i in range(n):
            a.src[i] = src_a[i]
            a.dst[i] = dst_a[i]
            a.row_bytes[i] = rb_a[i]
        a.capacity_rows = cap
        a.near_rel = float(near_rel)
        if rule not in RULES:
            raise OccamError(OCCAM_ERR_INVALID_ARG, f"rule must be one of {sorted(RULES)}")
        a.rule = RULES[rule]
        if rule == "budget":
            if budget is None:
                raise OccamError(OCCAM_ERR_INVALID_ARG, "rule 'budget' needs a budget tensor")
            budget = _dev_tensor(budget, torch.int32, "budget")
            if budget.numel() != B:
                raise OccamError(OCCAM_ERR_INVALID_ARG, "budget must have one entry per sample")
            self.keep_alive.append(budget)
            a.budget = _ptr(budget)
        self.args = a
        self.cout = CPruneOut(*[_ptr(o.get(k)) for k in
                                ("keep2", "out_index", "count_vis", "count_out", "out_off", "keep1", "s1", "ref1",
                                 "s2", "ref2", "n1_vis", "n_eff", "near1", "near2")])
        self.capacity = cap

    def __call__(self, stream=None) -> dict:
        if self.k2_stage is not None:
            _check(library().occam_prune_staged(ctypes.byref(self.args), ctypes.byref(self.cout),
                                                _ptr(self.k2_stage),
                                                self.k2_stage.numel() * self.k2_stage.element_size(),
                                                _ptr(self.ws), self.ws.numel(), _stream(stream)),
                   "occam_prune_staged")
            return self.out
        _check(library().occam_prune(ctypes.byref(self.args), ctypes.byref(self.cout), _ptr(self.ws),
                                     self.ws.numel(), _stream(stream)), "occam_prune")
        return self.out

    TRACE_NAMES = ("stage1", "stage1_finalize", "s1_list_plan", "stage2_fused", "stage2_twopass", "scan", "gather")

    def traced(self, events, stream=None) -> dict:
        """As __call__, recording ``events`` (torch.cuda.Event, enable_timing) between the kernels."""
        if self.k2_stage is not None:
            raise OccamError(OCCAM_ERR_UNSUPPORTED, "traced calls take device inputs")
        arr = (_p * len(events))(*[e.cuda_event for e in events])
        _check(library().occam_prune_traced(ctypes.byref(self.args), ctypes.byref(self.cout), _ptr(self.ws),
                                            self.ws.numel(), _stream(stream), arr, len(events)),
               "occam_prune_traced")
        return self.out

    def status(self, stream=None) -> int:
        return occam_get_status(self.ws, stream)


def occam_prune(layout: BatchLayout, stage1: dict, stage2: dict, lambda1: float, lambda2: float,
                keep_registers: bool = True, gather=(), capacity_rows: int | None = None,
                want=PruneCall.OPTIONAL, ws=None, stream=None, host_inputs: bool = False,
                rule: str = "register", budget=None, near_rel: float = 0.0) -> dict:
    """One fused prune call; returns the output tensors and the gathered rows.
    With host_inputs, K2 and the gather tensors may be pinned host tensors
    (occam_prune_staged). rule / budget select the rule variant (PruneCall);
    want may add "near1" / "near2" (PruneCall.NEAR), with band near_rel."""
    call = PruneCall(layout, stage1, stage2, lambda1, lambda2, keep_registers, gather, capacity_rows, want, ws,
                     host_inputs, rule, budget, near_rel)
    out = dict(call(stream))
    out["gathered"] = call.gathered
    out["ws"] = call.ws
    return out
