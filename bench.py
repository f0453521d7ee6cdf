"""Throughput of the OccamToken prune path (score -> threshold -> compact).

One step = one fused occam_prune call (Stage-I [CLS] scores and threshold,
Stage-II text scores and threshold, compaction and gather of the kept hidden /
K / V rows) over one batch of the LLaVA-NeXT-shaped workload: 64 images x
5 crops x (576 visual + 4 register rows), text lengths 16..256, synthetic
seeded inputs resident in HBM (about 5 GB per step: larger than L2, so no
flush is needed between steps).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints one JSON line. With N > 1 (torchrun) every rank runs an independent
replica of the batch ("replicas only": samples are independent and nothing
is exchanged); value = images processed by all ranks / max-over-ranks time.
The reference arm (--impl reference) times the CPU oracle, as it stands, on a
bounded sample of the same workload on this machine's host cores.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

WORKLOAD = "llavanext_b64"
METRIC = "pruned images/sec (score+threshold+compact) at 1 GB300; achieved HBM GB/s vs peak"
UNIT = "images/s"
FALLBACK_HBM_GBS = 6800.0
SPEC_HBM_GBS = 8000.0
KERNEL_SOURCES = {
    "stage1": "stage1.cu", "stage1_finalize": "stage1.cu", "s1_list_plan": "stage2.cu",
    "stage2_fused": "stage2_tc.cu", "stage2_twopass": ("stage2.cu", "stage2_scores_tc.cu"), "scan": "compact.cu",
    "gather": "compact.cu",
}


# ----------------------------------------------------------------------------- helpers

def _dist():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d.get("hbm_gbs", FALLBACK_HBM_GBS)), "measured"
    return FALLBACK_HBM_GBS, "fallback"


def _peak_tflops_sustained():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return float(json.load(f).get("bf16_tflops_sustained", 1700.0))
    return 1700.0


class ClockSampler:
    """Samples SM clocks / throttle reasons with nvidia-smi while running."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict | None:
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def _traffic_from_profiles(kernel: str):
    """dram bytes per launch of `kernel` from a committed ncu summary, if the
    kernel source is unchanged since it was taken; else None."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{WORKLOAD}.md")
    if not os.path.exists(path):
        return None
    txt = open(path).read()
    vals = {}
    for line in txt.splitlines():
        line = line.strip().strip("`")
        if "=" in line and line.split("=")[0].strip() in ("dram_bytes_per_launch", "source_sha"):
            k, v = line.split("=", 1)
            vals[k.strip()] = v.strip()
    if "dram_bytes_per_launch" not in vals or "source_sha" not in vals:
        return None
    files = KERNEL_SOURCES[kernel]
    files = (files,) if isinstance(files, str) else files
    h = hashlib.sha256()
    for f in files:  # a kernel built from several sources hashes their concatenation
        h.update(open(os.path.join(ROOT, "paper_2605_29657_gb300", "csrc", f), "rb").read())
    sha = h.hexdigest()[:16]
    if sha != vals["source_sha"]:
        return None
    return float(vals["dram_bytes_per_launch"])


def algorithmic_bytes(meta: dict, n1_total: int, kept_total: int) -> dict:
    """Bytes each kernel must move per launch (what the method needs, not the
    dense work it avoids), from this run's actual S1 sizes and kept rows."""
    rows, S, T = meta["total_rows"], meta["S_tot"], meta["total_text"]
    H1, d1, H2, d2, hid = meta["H1"], meta["d1"], meta["H2"], meta["d2"], meta["hidden"]
    k1row = H1 * d1 * 2
    H2kv = meta.get("H2kv", H2)          # key heads (fewer than H2 under grouped-query attention)
    k2row = H2kv * d2 * 2                # one K2 / K_text row
    qrow = H2 * d2 * 2                   # one Q_text row
    hrow = hid * 2                       # bytes of one hidden / V row (bf16)
    cls = meta["stage1"] == "cls"
    b = {}
    if cls:
        b["stage1"] = rows * k1row + S * k1row + rows * H1 * 4           # K1 once, q_cls, logits write
        b["stage1_finalize"] = rows * (H1 * 4 + 4 + 4 + 1 + 1 + 4) + S * k1row  # logits, s1 + s2 zero, role, keep1, list; q/k_cls
    else:
        b["stage1"] = 2 * rows * 2 * k1row                               # Q1 and K1 in each of the two passes
        b["stage1_finalize"] = rows * (4 + 1 + 1 + 4)                   # s1, role, keep1, list
    b["s1_list_plan"] = 0                                            # planned inside the finalize kernel
    b["stage2_fused"] = n1_total * k2row + T * (qrow + k2row)          # S1 keys once, Q + K_text
    b["stage2_twopass"] = 2 * n1_total * k2row + T * (2 * qrow + k2row) + 2 * T * H2 * 8  # both passes
    b["scan"] = rows * (1 + 1 + 4 + 1) + kept_total * 4              # keep1, role, s2, keep2, out_index
    b["gather"] = kept_total * 2 * (2 * hrow + k2row)                # read + write hidden, K, V rows
    # whole step, each byte once: K1, S1 keys, text Q/K, hidden+V of kept rows
    # (their K rows were read for scoring), writes of the 3 gathered rows
    stage1_in = rows * k1row + 2 * S * k1row if cls else 2 * rows * k1row   # K1 (+ q/k_cls) or Q1 + K1, once
    step = (stage1_in + n1_total * k2row + T * (qrow + k2row)
            + kept_total * (2 * hrow) + kept_total * (2 * hrow + k2row) + rows + kept_total * 4)
    b["step"] = step
    return b


def _kernel_stats(occ, events):
    """Per-kernel interval means (ms) and, per kernel, the spread over the
    traced calls (min, max, standard deviation)."""
    mean, spread = {}, {}
    for j, name in enumerate(occ.PruneCall.TRACE_NAMES):
        xs = [evs[j].elapsed_time(evs[j + 1]) for evs in events]
        mean[name] = float(np.mean(xs))
        spread[name] = {"min": float(np.min(xs)), "max": float(np.max(xs)), "std": float(np.std(xs)), "n": len(xs)}
    return mean, spread


def mutual_stage1_flops(meta: dict) -> float:
    """Multiply-add FLOPs of the mutual Stage I (Sec. 3.4, Eq. 6): per
    segment of n rows, two passes of n x n logits per head over d1 dims."""
    seg = np.diff(np.asarray(meta["seg_off_host"], dtype=np.int64)).astype(np.float64)
    return float(2 * np.sum(2.0 * seg * seg * meta["H1"] * meta["d1"]))


def measure_workload(occ, name: str, dev, steps: int, warmup: int, l2_flush: bool = False, n_traced: int = 20,
                     peak_gbs: float = FALLBACK_HBM_GBS, peak_tflops: float = 0.0) -> dict:
    """One workload, one occam_prune call at a time: `steps` replays of the
    call's CUDA graph timed with CUDA events (with l2_flush, a 256 MB buffer
    is written before every step and each step is timed alone), then
    `n_traced` eager calls recording per-kernel events."""
    import torch
    from synth import get_config, make_batch

    w = get_config(name)
    batch = make_batch(w, device=dev, seed=w.seed)
    meta = batch["meta"]
    layout = occ.BatchLayout.from_batch(batch, dev)
    cls = w.stage1 == "cls"
    st1 = (dict(mode="cls", q=batch["q_cls"], k_cls=batch["k_cls"], K1=batch["K1"]) if cls else
           dict(mode="mutual", q=batch["Q1"], K1=batch["K1"]))
    call = occ.PruneCall(layout, st1, dict(Q_text=batch["Q_text"], K_text=batch["K_text"], K2=batch["K2"]),
                         w.lambda1, w.lambda2, keep_registers=True,
                         gather=(batch["hidden"], batch["K2"].view(batch["K2"].shape[0], -1), batch["V"]))
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        call()
    call()
    torch.cuda.synchronize()
    if call.status() != 0:
        raise RuntimeError(f"device status {call.status()} on {name}")
    kernels = occ.occam_last_call_kernels()
    out = call.out
    n1_total = int(out["n1_vis"].sum().item()) + int(meta["regs_per_seg"] * meta["S_tot"])
    kept_total = int(out["out_off"][-1].item())
    bytes_ = algorithmic_bytes(meta, n1_total, kept_total)
    want = {k: v.clone() for k, v in out.items()}
    cap = torch.cuda.Stream(device=dev)
    cap.wait_stream(stream)
    with torch.cuda.stream(cap):
        call(cap)
    stream.wait_stream(cap)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        call()
    g.replay()
    torch.cuda.synchronize()
    for k, v in want.items():
        same = torch.equal(v[:kept_total], out[k][:kept_total]) if k == "out_index" else torch.equal(v, out[k])
        if not same:
            raise RuntimeError(f"{name}: a graph replay differs from the eager call in {k}")
    if l2_flush:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
        for i, (a, b) in enumerate(ev):
            flush.fill_(i & 255)
            a.record(stream)
            g.replay()
            b.record(stream)
        torch.cuda.synchronize()
        ms = float(sum(a.elapsed_time(b) for a, b in ev))
        del flush
    else:
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(steps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        ms = a.elapsed_time(b)
    nk = len(occ.PruneCall.TRACE_NAMES) + 1
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(nk)] for _ in range(n_traced)]
    for evs in events:  # torch creates an event's CUDA handle on its first record
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize()
    for evs in events:
        call.traced(evs, stream)
    torch.cuda.synchronize()
    if call.status() != 0:
        raise RuntimeError(f"device status {call.status()} on {name} after timing")
    per_kernel, spread = _kernel_stats(occ, events)
    dom = max(per_kernel, key=per_kernel.get)
    step_ms = ms / steps
    res = {
        "ms_per_step": step_ms, "images_per_s": meta["B"] / (step_ms / 1e3), "steps": steps,
        "l2": "a 256 MB buffer written before every step (L2 flushed)" if l2_flush else
              ("no flush: inputs " + ("larger" if bytes_["step"] > (128 << 20) else "smaller") + " than L2"),
        "mean_n1_vis": float(out["n1_vis"].float().mean().item()),
        "mean_count_vis": float(out["count_vis"].float().mean().item()),
        "algorithmic_bytes_per_step": bytes_["step"],
        "step_frac_of_measured_hbm": bytes_["step"] / (step_ms / 1e3) / 1e9 / peak_gbs,
        "dominant_interval": dom, "dominant_ms": per_kernel[dom], "dominant_ms_spread": spread[dom],
        "kernels_per_step": kernels, "per_kernel_ms": per_kernel,
    }
    if cls or dom != "stage1":
        res["dominant_frac_of_measured_hbm"] = bytes_[dom] / (per_kernel[dom] / 1e3) / 1e9 / peak_gbs
    if not cls:
        fl = mutual_stage1_flops(meta)
        tf = fl / (per_kernel["stage1"] / 1e3) / 1e12
        res["stage1_mutual"] = {"flops": fl, "achieved_tflops": tf, "peak_tflops": peak_tflops,
                                "frac": tf / peak_tflops if peak_tflops else None,
                                "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained",
                                "note": "multiply-add FLOPs of both passes (2 n^2 H1 d1 each per segment)"}
    del call, g, batch, out, want
    torch.cuda.empty_cache()
    return res


def aggregate(ms_local: float, images_local: int, device=None):
    """Max of the timed milliseconds and sum of the images over all ranks
    (replicas: nothing else is exchanged)."""
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms_local], dtype=torch.float64, device=device)
    n = torch.tensor([images_local], dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n.item())


# ----------------------------------------------------------------------------- CPU oracle (baseline / reference arm)

def _oracle_worker(args):
    """Generates its own samples of the workload (untimed), then times the
    oracle on them. Runs in a spawned process with single-threaded BLAS."""
    seeds, = args
    sys.path.insert(0, ROOT)
    from oracle import occam_oracle as O
    from synth import get_config, make_batch
    w = get_config(WORKLOAD)
    one = get_config(WORKLOAD, B=1)
    batches = [make_batch(one, seed=int(s)) for s in seeds]
    t0 = time.perf_counter()
    for b in batches:
        O.prune(b, w.lambda1, w.lambda2)
    return time.perf_counter() - t0, len(batches)


def oracle_throughput(n_workers: int, samples_per_worker: int, seed0: int, pool=None) -> dict:
    import multiprocessing as mp
    own = pool is None
    if own:
        pool = _make_pool(n_workers)
    jobs = [([seed0 + 1000 + i * samples_per_worker + k for k in range(samples_per_worker)],)
            for i in range(n_workers)]
    res = pool.map(_oracle_worker, jobs)
    if own:
        pool.close()
        pool.join()
    wall = max(t for t, _ in res)
    n = sum(k for _, k in res)
    del mp
    return {"value": n / wall, "unit": UNIT, "cores": n_workers, "kind": "oracle",
            "sample": f"{n} samples of the {WORKLOAD} workload (batch of one each), "
                      f"{samples_per_worker} per worker on {n_workers} single-threaded workers; "
                      f"value = samples / slowest worker's oracle time",
            "seconds": wall, "cpu_seconds": sum(t for t, _ in res)}


def _make_pool(n):
    import multiprocessing as mp
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[k] = "1"
    return mp.get_context("spawn").Pool(n)


# ----------------------------------------------------------------------------- GPU arm

def run_ours(args, rank, world, local):
    import torch
    import torch.distributed as dist

    import paper_2605_29657_gb300 as occ
    from synth import get_config, make_batch

    # host-core oracle pool first: spawn, before the first GPU call; one
    # single-threaded worker per host core
    n_workers = os.cpu_count() or 1
    pool = _make_pool(n_workers) if (rank == 0 and not args.no_cpu_baseline) else None

    occ.occam_set_stage2_route({"auto": occ.OCCAM_ROUTE_AUTO, "narrow": occ.OCCAM_ROUTE_NARROW,
                                "twopass": occ.OCCAM_ROUTE_TWOPASS}[args.route])
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    w = get_config(WORKLOAD)
    if args.kv_heads:
        from dataclasses import replace
        w = replace(w, H2kv=args.kv_heads)   # a grouped-query LLM layer of the same shape
    batch = make_batch(w, device=dev, seed=w.seed + 0)  # every rank: its own replica of the batch
    meta = batch["meta"]
    layout = occ.BatchLayout.from_batch(batch, dev)
    gather = (batch["hidden"], batch["K2"].view(batch["K2"].shape[0], -1), batch["V"])
    cls = w.stage1 == "cls"
    stage1_of = ((lambda t: dict(mode="cls", q=t["q_cls"], k_cls=t["k_cls"], K1=t["K1"])) if cls else
                 (lambda t: dict(mode="mutual", q=t["Q1"], K1=t["K1"])))
    # `inflight` prune calls in flight at once, each with its own copy of the
    # inputs, workspace and outputs, on its own stream: consecutive steps
    # overlap on the GPU as consecutive batches of a serving loop would. The
    # copies keep the calls from sharing L2 hits on one set of inputs.
    inflight = max(1, args.inflight)
    input_names = ("q_cls", "k_cls", "Q1", "K1", "Q_text", "K_text", "K2", "hidden", "V")
    sets = [batch] + [{k: (v.clone() if k in input_names else v) for k, v in batch.items()}
                      for _ in range(inflight - 1)]

    def make_call(t):
        return occ.PruneCall(layout, stage1_of(t), dict(Q_text=t["Q_text"], K_text=t["K_text"], K2=t["K2"]),
                             w.lambda1, w.lambda2, keep_registers=True,
                             gather=(t["hidden"], t["K2"].view(t["K2"].shape[0], -1), t["V"]))

    calls = [make_call(t) for t in sets]
    call = calls[0]
    stream = torch.cuda.current_stream()
    streams = [stream] if inflight == 1 else [torch.cuda.Stream(device=dev) for _ in range(inflight)]
    nk = len(occ.PruneCall.TRACE_NAMES) + 1

    for c, s_ in zip(calls, streams):
        for _ in range(args.warmup):
            c(s_)
    torch.cuda.synchronize()
    for c in calls:
        st = c.status()
        if st != 0:
            raise RuntimeError(f"device status {st} after warm-up")
    out = call.out
    call()                                         # an eager call, to count the kernels it launches
    torch.cuda.synchronize()
    kernels_per_step = occ.occam_last_call_kernels()
    n1_total = int(out["n1_vis"].sum().item()) + int(meta["regs_per_seg"] * meta["S_tot"])  # registers are in S1
    kept_total = int(out["out_off"][-1].item())
    bytes_ = algorithmic_bytes(meta, n1_total, kept_total)
    want = {k: v.clone() for k, v in call.out.items()}
    # near-threshold rows of the two tests (band 1e-5), from one more eager
    # call with the flags requested (outside the timed region, no gather)
    ncall = occ.PruneCall(layout, stage1_of(batch),
                          dict(Q_text=batch["Q_text"], K_text=batch["K_text"], K2=batch["K2"]),
                          w.lambda1, w.lambda2, keep_registers=True,
                          want=occ.PruneCall.OPTIONAL + occ.PruneCall.NEAR, ws=call.ws)
    ncall()
    torch.cuda.synchronize()
    if ncall.status() != 0:
        raise RuntimeError("device status after the near-threshold call")
    near_rows = {"stage1": int(ncall.out["near1"].sum().item()), "stage2": int(ncall.out["near2"].sum().item()),
                 "band": "|s - tau| <= 1e-5 |tau| (visual rows; S1 rows for Stage II)"}
    del ncall

    def same_as_first(c, what):
        for k, v in want.items():
            if k == "out_index":
                ok = torch.equal(v[:kept_total], c.out[k][:kept_total])
            else:
                ok = torch.equal(v, c.out[k])
            if not ok:
                raise RuntimeError(f"{what} differs from the first eager call in {k}")

    for c in calls[1:]:
        same_as_first(c, "a second in-flight call (same inputs)")

    # each call captured once as a CUDA graph: the timed steps replay them
    # (one replay = one whole occam_prune call, every kernel), which removes
    # the host's per-call launch work; replays must equal the eager call
    graphs = None
    if not args.no_graph:
        graphs = []
        for c in calls:
            cap_stream = torch.cuda.Stream(device=dev)
            cap_stream.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(cap_stream):
                c(cap_stream)
            torch.cuda.current_stream().wait_stream(cap_stream)
            torch.cuda.synchronize()
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                c()
            g.replay()
            torch.cuda.synchronize()
            same_as_first(c, "a graph replay")
            graphs.append(g)

    # per-kernel events come from eager calls made one at a time on one
    # stream after the timed region (so a kernel's interval is its own, not
    # shared with another call's kernels, and `value` is untouched)
    n_traced = max(20, min(args.steps // 5, 200))
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(nk)] for _ in range(n_traced)]
    for evs in events:  # torch creates an event's CUDA handle on its first record
        for e in evs:
            e.record(stream)
    torch.cuda.synchronize()

    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for s_ in streams[1:]:
        s_.wait_event(t_start)
    for i in range(args.steps):
        j = i % inflight
        with torch.cuda.stream(streams[j]):
            if graphs is not None:
                graphs[j].replay()
            else:
                calls[j]()
    for s_ in streams[1:]:
        stream.wait_stream(s_)
    t_end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = sampler.stop()
    ms = t_start.elapsed_time(t_end)
    for c in calls:
        st = c.status()
        if st != 0:
            raise RuntimeError(f"device status {st} after the timed steps")
        same_as_first(c, "a call after the timed steps")
    for evs in events:
        calls[0].traced(evs, stream)
    torch.cuda.synchronize()
    per_kernel, per_kernel_spread = _kernel_stats(occ, events)

    ms_max, images = aggregate(ms, meta["B"] * args.steps, dev)
    value = images / (ms_max / 1e3)

    # ---- end to end through the public API with host buffers: every input
    # starts in pinned host memory each step. The scoring inputs (q/k_cls,
    # K1, Q_text, K_text) are copied to the device; K2, hidden and V stay on
    # the host and occam_prune_staged reads only what the method needs from
    # them across the host link (the S1 rows of K2, the kept rows of hidden
    # and V; the kept rows of K2 come from its staged S1 rows). The results
    # (counts, offsets, indices) are read back.
    e2e = None
    if not args.no_e2e:
        copy_names = (["q_cls", "k_cls"] if cls else ["Q1"]) + ["K1", "Q_text", "K_text"]
        host = {k: batch[k].cpu().pin_memory() for k in copy_names + ["K2", "hidden", "V"]}
        K2h = host["K2"]
        res_names = ["count_vis", "count_out", "out_off", "out_index"]
        # two sets of device inputs and calls: the next step's host->device
        # copies (on a copy stream) run while the current step computes
        nset = 2
        dins, hcalls, res_host = [], [], []
        for _ in range(nset):
            d = {k: torch.empty_like(batch[k]) for k in copy_names}
            dins.append(d)
            hcalls.append(occ.PruneCall(layout, stage1_of(d),
                                        dict(Q_text=d["Q_text"], K_text=d["K_text"], K2=K2h),
                                        w.lambda1, w.lambda2, keep_registers=True,
                                        gather=(host["hidden"], K2h.view(K2h.shape[0], -1), host["V"]),
                                        host_inputs=True))
            res_host.append({k: torch.empty_like(hcalls[-1].out[k], device="cpu").pin_memory() for k in res_names})
        copy_stream = torch.cuda.Stream(device=dev)
        copied = [torch.cuda.Event() for _ in range(nset)]
        done = [torch.cuda.Event() for _ in range(nset)]
        copied_bytes = sum(host[k].numel() * host[k].element_size() for k in copy_names)
        k2row = meta.get("H2kv", meta["H2"]) * meta["d2"] * 2
        # the kept rows of K2 are read from the staged S1 rows on the device
        kept_row = sum(host[k][0].numel() * host[k].element_size() for k in ("hidden", "V"))
        in_place = n1_total * k2row + kept_total * kept_row
        d2h = sum(t.numel() * t.element_size() for t in res_host[0].values())

        def e2e_step(i):
            s = i % nset
            with torch.cuda.stream(copy_stream):
                copy_stream.wait_event(done[s])  # the set's previous step is finished
                for k in copy_names:
                    dins[s][k].copy_(host[k], non_blocking=True)
                copied[s].record(copy_stream)
            stream.wait_event(copied[s])
            hcalls[s](stream)
            for k in res_names:
                res_host[s][k].copy_(hcalls[s].out[k], non_blocking=True)
            done[s].record(stream)

        for i in range(2 * nset):
            e2e_step(i)
        torch.cuda.synchronize()
        for hc, rh in zip(hcalls, res_host):
            if hc.status() != 0:
                raise RuntimeError("device status after the host-input warm-up")
            # the host-input call must reproduce the device-input call exactly
            for k in ("count_vis", "count_out", "out_off"):
                if not torch.equal(rh[k], call.out[k].cpu()):
                    raise RuntimeError(f"host-input call differs from the device-input call in {k}")
            if not torch.equal(rh["out_index"][:kept_total], call.out["out_index"][:kept_total].cpu()):
                raise RuntimeError("host-input call differs from the device-input call in out_index")
        e_steps = max(20, min(50, args.steps // 20))
        # the host link's own rate: the largest scoring input copied host ->
        # device by the copy engine (best of 3), before and after the timed blocks
        big = max(copy_names, key=lambda k: host[k].numel() * host[k].element_size())
        big_bytes = host[big].numel() * host[big].element_size()

        def link_rate():
            l0 = torch.cuda.Event(enable_timing=True)
            l1 = torch.cuda.Event(enable_timing=True)
            best = None
            for _ in range(3):
                l0.record(copy_stream)
                with torch.cuda.stream(copy_stream):
                    dins[0][big].copy_(host[big], non_blocking=True)
                l1.record(copy_stream)
                torch.cuda.synchronize()
                t = l0.elapsed_time(l1)
                best = t if best is None else min(best, t)
            return big_bytes / (best / 1e3) / 1e9

        link_before = link_rate()
        # three timed blocks of e_steps steps; the host (its memory and link)
        # is shared with other jobs, so the median block is reported, with all three
        blocks = []
        for _ in range(3):
            if world > 1:
                dist.barrier()
            a = torch.cuda.Event(enable_timing=True)
            z = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            copy_stream.wait_event(a)
            for i in range(e_steps):
                e2e_step(i)
            z.record(stream)
            torch.cuda.synchronize()
            blocks.append(aggregate(a.elapsed_time(z), meta["B"] * e_steps, dev))
        link_after = link_rate()
        ems, e_images = sorted(blocks, key=lambda bl: bl[0])[1]
        link_gbs = max(link_before, link_after)
        step_gbs = (copied_bytes + in_place) / (ems / e_steps / 1e3) / 1e9
        e2e = {"value": e_images / (ems / 1e3), "unit": UNIT,
               "blocks": [bi / (bm / 1e3) for bm, bi in blocks],
               "host_link": {"h2d_gbs": link_gbs, "before": link_before, "after": link_after, "bytes": int(big_bytes),
                             "tensor": big,
                             "how": "copy-engine host->device copy from pinned memory, best of 3, before and after "
                                    "the timed blocks (the larger is h2d_gbs)"},
               "h2d_gbs_per_step": step_gbs, "frac_of_host_link": step_gbs / link_gbs,
               "h2d_bytes_per_step": int(copied_bytes + in_place), "d2h_bytes_per_step": int(d2h),
               "steps": e_steps, "timed_blocks": 3, "h2d_copied_bytes_per_step": int(copied_bytes),
               "h2d_read_in_place_bytes_per_step": int(in_place),
               "inputs": f"pinned host memory; {', '.join(copy_names)} copied each step (two device "
                         "input sets, the next step's copies overlapping the current step); K2, hidden, V "
                         "read in place (S1 rows of K2, kept rows of hidden and V)"}

    # ---- the rows beyond the pruning path, timed on this workload's tensors
    # (outside the step; not part of `value`)
    next_rows = None
    if not args.no_next:
        def timed(fn, reps=20):
            for _ in range(3):
                fn()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(reps):
                fn()
            e1.record(stream)
            torch.cuda.synchronize()
            return e0.elapsed_time(e1) / reps

        K_tar = int(round(float(out["count_vis"].float().mean().item()) * meta["B"]))
        lam_ms = timed(lambda: occ.occam_calibrate_lambda2(layout, out["s2"], out["ref2"], out["keep1"], K_tar,
                                                             ws=call.ws))
        lam, ncand = occ.occam_calibrate_lambda2(layout, out["s2"], out["ref2"], out["keep1"], K_tar, ws=call.ws)
        k_reg = torch.tensor([7, 100, 511, 1000, 2047, 2048, 3000, 3333, 4000, 4095], dtype=torch.int32,
                             device=dev)
        h_copy = batch["hidden"].clone()
        reg_ms = timed(lambda: occ.occam_construct_registers(layout, h_copy, k_reg, ws=call.ws))
        del h_copy
        next_rows = {
            "lambda2_budget": {"ms": lam_ms, "target_rows": K_tar, "candidates": int(ncand.item()),
                               "lambda2": float(lam.item()), "calibrated_lambda2": w.lambda2,
                               "how": "radix select of the K-th largest s2/ref2 over the step's S1 rows (11-bit digits, grid-wide histograms; one pass of kept counts for the fp32 product rule)"},
            "register_construction": {"ms": reg_ms, "rows": meta["total_rows"], "channels": 10,
                                      "how": "in place on hidden [rows, 4096] bf16, per segment"},
            "n_eff": "computed in the Stage-I finalize of every timed step ([CLS] mode, optional output)",
        }
        # the component ablation's rule variants as whole prune steps on the
        # same tensors. Mean threshold: lambdas scaled by the step's average
        # register / mean reference ratio (thresholds matched on average).
        # Fixed budget: every sample keeps the step's average count_vis.
        ref1m = occ.occam_mean_reference(layout, out["s1"], occ.OCCAM_REF_SEGMENT)
        ref2m = occ.occam_mean_reference(layout, out["s2"], occ.OCCAM_REF_SAMPLE, prev_keep=out["keep1"])
        r1 = float((out["ref1"] / ref1m.clamp_min(1e-30)).mean().item())
        r2 = float((out["ref2"] / ref2m.clamp_min(1e-30)).mean().item())
        avg_budget = int(round(float(out["count_vis"].float().mean().item())))
        budget = torch.full((meta["B"],), avg_budget, dtype=torch.int32, device=dev)
        variants = {}
        for rule, l1, l2, bud in (("mean", w.lambda1 * r1, w.lambda2 * r2, None),
                                  ("budget", w.lambda1, w.lambda2, budget)):
            vcall = occ.PruneCall(layout, stage1_of(batch),
                                  dict(Q_text=batch["Q_text"], K_text=batch["K_text"], K2=batch["K2"]),
                                  l1, l2, keep_registers=True, gather=gather, rule=rule, budget=bud,
                                  ws=call.ws)
            v_ms = timed(lambda: vcall())
            if vcall.status() != 0:
                raise RuntimeError(f"device status after the {rule} rule")
            variants[rule] = {"ms_per_step": v_ms, "images_per_s": meta["B"] / (v_ms / 1e3),
                              "kept_rows": int(vcall.out["out_off"][-1].item()),
                              "lambda1": l1, "lambda2": l2 if rule == "mean" else None,
                              "budget_per_sample": avg_budget if rule == "budget" else None}
            del vcall
        next_rows["rule_variants"] = variants

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return None

    peak, peak_kind = _peaks()
    # the other workloads of the configuration list, one call at a time
    # (parity-test shapes, reported beside the headline; not part of `value`)
    workloads = None
    used_graph = graphs is not None
    if not args.no_workloads:
        del sets, calls, graphs
        torch.cuda.empty_cache()
        wsteps = max(50, min(300, args.steps // 4))
        workloads = {}
        for nm in ("llava15_b1", "llavanext_b8", "qwen3vl_b32", "video_b4"):
            workloads[nm] = measure_workload(occ, nm, dev, wsteps, 5, peak_gbs=peak,
                                             peak_tflops=_peak_tflops_sustained())
        for nm in ("llava15_b1", "llavanext_b8"):
            workloads[nm + "_l2flush"] = measure_workload(occ, nm, dev, wsteps, 5, l2_flush=True, peak_gbs=peak)
    dom = max(per_kernel, key=per_kernel.get)
    achieved = bytes_[dom] / (per_kernel[dom] / 1e3) / 1e9
    traffic = _traffic_from_profiles(dom)
    roofline = {"bound": "hbm", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "GB/s",
                "frac": achieved / peak, "traffic": traffic, "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)"
                if peak_kind == "measured" else "fallback 6.8 TB/s",
                "algorithmic_bytes_per_launch": bytes_[dom], "avg_launch_ms": per_kernel[dom]}
    roofline["timing"] = (f"avg_launch_ms from CUDA events around the kernel in {n_traced} eager calls made one at "
                          "a time after the timed region (outside `value`)")
    roofline["launch_ms_spread"] = per_kernel_spread[dom]
    step_ms = ms_max / args.steps
    step_gbs = bytes_["step"] / (step_ms / 1e3) / 1e9
    cpu = None
    if pool is not None:
        cpu = oracle_throughput(n_workers, 10, 0, pool=pool)
        pool.close()
        pool.join()
        one = oracle_throughput(1, 8, 50_000)   # the same oracle on one core, alone
        cpu["single_thread"] = {"value": one["value"], "unit": UNIT, "cores": 1, "sample": one["sample"]}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {
            "workload": WORKLOAD, "B": meta["B"], "crops": meta["segs_per_sample"],
            "visual_per_crop": (w.vis[1] if w.vis[0] == "fixed" else f"{w.vis[1]}..{w.vis[2]} (step {w.vis[3]})"),
            "registers_per_crop": meta["regs_per_seg"],
            "text_tokens": (str(w.M[1]) if w.M[0] == "fixed" else f"{w.M[1]}..{w.M[2]} (uniform)"),
            "H1xd1": f"{meta['H1']}x{meta['d1']}", "H2xd2": f"{meta['H2']}x{meta['d2']}", "hidden": meta["hidden"],
            "kv_heads": meta.get("H2kv", meta["H2"]),
            "lambda1": w.lambda1, "lambda2": w.lambda2, "accumulate": "fp32",
            "parallelism": "replicas" if world > 1 else "single",
            "l2": "inputs larger than L2 (about 5 GB resident per step); no flush",
            "launch": (f"{inflight} occam_prune calls in flight on {inflight} streams, each with its own copy of "
                       "the inputs, workspace and outputs; a step replays one call's CUDA graph (every kernel of "
                       f"the call); per-kernel events from {n_traced} eager calls after the timed region")
                      if used_graph else
                      f"{inflight} eager occam_prune calls in flight on {inflight} streams "
                      f"(per-kernel events from {n_traced} eager calls after the timed region)",
            "inflight": inflight,
            "mean_n1_vis": float(out["n1_vis"].float().mean().item()),
            "mean_count_vis": float(out["count_vis"].float().mean().item()),
            "kept_rows_per_step": kept_total,
            "near_threshold_rows": near_rows,
            "algorithmic_bytes_per_step": bytes_["step"],
            "step_algorithmic_GBps": step_gbs,
            "step_frac_of_measured_hbm": step_gbs / peak,
            "step_frac_of_8TBps": step_gbs / SPEC_HBM_GBS,
            "per_kernel_ms": per_kernel,
            "per_kernel_ms_spread": per_kernel_spread,
        },
        "roofline": roofline,
        "cpu_baseline": cpu,
        "e2e": e2e,
        # kernels per occam_prune call: Stage I (1 [CLS] / 2 mutual), finalize
        # (with the Stage-II plan), fused Stage II with 16-, 8- and 4-CTA
        # clusters, the two-pass Stage-II pair, scan, gather
        "gpu_launches": kernels_per_step * args.steps,
        "clocks": clocks,
        "next_rows": next_rows,
        "workloads": workloads,
    }
    if world > 1:
        dist.destroy_process_group()
    return line


# ----------------------------------------------------------------------------- reference arm

def run_reference(args, rank, world):
    if rank != 0:
        return None
    n_workers = os.cpu_count() or 1
    pool = _make_pool(n_workers)
    for i in range(args.warmup):
        oracle_throughput(n_workers, 1, 10_000 + i, pool=pool)
    vals, secs = [], 0.0
    n = 0
    for i in range(args.steps):
        r = oracle_throughput(n_workers, 1, 20_000 + i * n_workers, pool=pool)
        secs += r["seconds"]
        n += n_workers
    pool.close()
    pool.join()
    value = n / secs
    del vals
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "B_per_step": n_workers,
                   "note": "the CPU oracle (numpy float64) timed as it stands on this machine's host cores"},
        "cpu_baseline": {"kind": "oracle", "cores": n_workers, "value": value, "unit": UNIT,
                         "sample": f"each step: {n_workers} samples of the {WORKLOAD} workload, one per "
                                   f"single-threaded worker"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-graph", action="store_true", help="time eager calls instead of a captured CUDA graph")
    ap.add_argument("--kv-heads", type=int, default=0,
                    help="key / value heads of the LLM layer (grouped-query variant; 0: one per query head)")
    ap.add_argument("--inflight", type=int, default=3,
                    help="prune calls in flight at once (own inputs, workspace, outputs and stream each)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-next", action="store_true", help="skip timing the rows beyond the pruning path")
    ap.add_argument("--no-workloads", action="store_true", help="skip timing the other four workloads")
    ap.add_argument("--route", default="auto", choices=["auto", "narrow", "twopass"],
                    help="Stage-II routing (diagnostics; auto is the library default)")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="synthetic workload to time (default: the LLaVA-NeXT batch-64 throughput workload)")
    args = ap.parse_args()
    globals()["WORKLOAD"] = args.workload
    if args.warmup < 3:
        args.warmup = 3
    rank, world, local = _dist()
    if args.impl == "reference":
        line = run_reference(args, rank, world)
    else:
        import paper_2605_29657_gb300.build as pb
        pb.build()
        line = run_ours(args, rank, world, local)
    if line is not None and rank == 0:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
