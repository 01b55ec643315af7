"""Throughput of the pooled embedding-bag forward + de-duplicated backward on GB300.

One step = the whole hot path on one batch: forward gather-pool, then the
backward (key generation, radix sort, run-length pass, segmented reduce).
Prints one JSON line (rank 0). Defaults: 1 GPU, the 128 GB workload cfg5.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload cfg5]
  python bench.py --impl reference ...   # the fp64 CPU oracle on a bounded sample

Under torchrun every rank runs an independent replica (its own tables and
batches; no collective on the data path) and rank 0 reports the whole-job
throughput: all ranks' bytes over the slowest rank's time ("weak" scaling).
"""

from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2609_30656_gb300 import metrics, workloads as wl  # noqa: E402

METRIC = "embedding-bag fwd/bwd HBM GB/s and % of GB300 peak; rows gathered/sec"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


# ----------------------------------------------------------------------------- helpers

def measured_hbm_peak() -> tuple[float, str]:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def describe(w: wl.Workload) -> str:
    L = w.lengths
    if L.kind == "fixed":
        lens = f"every bag {int(L.mean)} long"
    elif L.kind == "poisson":
        lens = f"Poisson({L.mean:g}) lengths clipped to [{L.lo}, {L.hi}]"
    elif L.kind == "lognormal":
        lens = f"lognormal lengths (mean {L.mean:g}, max {L.hi})"
    else:
        lens = (f"{L.empty_frac:.0%} empty bags, others power law L^-{L.alpha:g} on "
                f"[{L.lo}, {L.hi}]")
    idx = "uniform indices" if w.zipf_alpha is None else f"Zipf({w.zipf_alpha:g}) indices"
    pool = ("weighted " if w.weighted else "") + ("mean" if w.mean else "sum")
    rows = (f"{w.num_tables} x {w.rows[0]:,} rows" if len(set(w.rows)) == 1
            else f"{w.num_tables} tables, {min(w.rows):,}..{max(w.rows):,} rows")
    dims = "/".join(str(d) for d in sorted(set(w.dims)))
    return (f"{w.name}: {rows} x dim {dims} {w.dtype}, batch {w.batch}, {lens}, {idx}, {pool} "
            f"pooling, forward + de-duplicated backward")


# The sources that compile each roofline kernel (and the build flags): the
# recorded DRAM traffic of a kernel holds while these are unchanged.
KERNEL_SOURCES = {
    "fwd.gather": ["tbe_internal.cuh", "tbe_forward.cuh", "tbe_forward_f32.cu", "tbe_forward_f16.cu",
                   "tbe_forward_bf16.cu", "tbe_launch.h", "../build.py"],
    "bwd.reduce": ["tbe_internal.cuh", "tbe_reduce.cuh", "tbe_reduce_f32.cu", "tbe_launch.h", "../build.py"],
}


def kernel_source_hash(kernel: str | None = None) -> str:
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_30656_gb300", "csrc")
    names = KERNEL_SOURCES[kernel] if kernel in KERNEL_SOURCES else sorted(os.listdir(csrc))
    for name in names:
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode())
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, if taken on this source."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except Exception:
        return None
    entry = rec.get(workload, {}).get(kernel)
    if not entry or entry.get("source_hash") != kernel_source_hash(kernel):
        return None
    return entry.get("bytes_per_launch")


class ClockSampler:
    """nvidia-smi clock / throttle sampling during the timed region."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200", "-i", str(self.index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        self.out = ""
        if self.proc is not None:
            time.sleep(0.3)
            self.proc.terminate()
            try:
                self.out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        for line in (self.out or "").splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != 7:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), float(parts[2]), parts[3:]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, _, flags in rows for i, fl in enumerate(flags)
                          if fl.lower().startswith("active")})
        loaded = [r for r in rows if r[2] > 200.0] or rows
        return {"sm_mhz": statistics.median(r[0] for r in loaded),
                "sm_max_mhz": max(r[1] for r in rows), "reasons": reasons,
                "samples": len(rows), "power_w_max": max(r[2] for r in rows)}


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def aggregate(local_ms: float, local_bytes: float, local_rows: float, world: int):
    """Max time and summed work over ranks (identity at world size 1)."""
    if world == 1 or not torch.distributed.is_initialized():
        return local_ms, local_bytes, local_rows
    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() and \
        torch.distributed.get_backend() == "nccl" else torch.device("cpu")
    t = torch.tensor([local_ms], dtype=torch.float64, device=dev)
    s = torch.tensor([local_bytes, local_rows], dtype=torch.float64, device=dev)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    torch.distributed.all_reduce(s, op=torch.distributed.ReduceOp.SUM)
    return float(t[0]), float(s[0]), float(s[1])


# ----------------------------------------------------------------------------- oracle leg

def _compact(tables, indices, offsets, weights, batch, tabs_idx):
    """Host copies of the rows touched by the chosen tables, indices renumbered."""
    host_tabs, host_ind, off_parts, w_parts = [], [], [], []
    lens = []
    for t in tabs_idx:
        s, e = int(offsets[t * batch]), int(offsets[(t + 1) * batch])
        idx = indices[s:e]
        uniq = torch.unique(idx)
        host_tabs.append(tables[t].index_select(0, uniq).cpu())
        host_ind.append(torch.searchsorted(uniq, idx).cpu())
        lens.append((offsets[t * batch + 1:(t + 1) * batch + 1] -
                     offsets[t * batch:(t + 1) * batch]).cpu())
        if weights is not None:
            w_parts.append(weights[s:e].cpu())
    L = torch.cat(lens)
    off = torch.zeros(L.numel() + 1, dtype=torch.int64)
    off[1:] = torch.cumsum(L, 0)
    ind = torch.cat(host_ind) if host_ind else torch.zeros(0, dtype=torch.int64)
    w = torch.cat(w_parts) if weights is not None else None
    return host_tabs, ind, off, w


def oracle_step(host_tabs, ind, off, w, go, batch, mean, threads):
    import numpy as np

    import oracle
    t0 = time.perf_counter()
    oracle.forward(host_tabs, batch, ind, off, weights=w, mean=mean, threads=threads)
    rows = np.array([t.shape[0] for t in host_tabs], np.int64)
    dims = np.array([t.shape[1] for t in host_tabs], np.int32)
    res = oracle.backward(rows, dims, batch, ind, off, go, weights=w, mean=mean, threads=threads)
    return time.perf_counter() - t0, res


def sample_problem(w, tables, batch0, go0, num_tables):
    tabs_idx = list(range(num_tables))
    host_tabs, ind, off, wt = _compact(tables, batch0.indices, batch0.offsets, batch0.weights,
                                       w.batch, tabs_idx)
    dims = [w.dims[t] for t in tabs_idx]
    cols = []
    for t in tabs_idx:
        d0 = sum(w.dims[:t])
        cols.append(go0[:, d0:d0 + w.dims[t]])
    go = torch.cat(cols, dim=1).cpu().contiguous()
    counts = metrics.batch_counts(dims, w.elem_bytes, w.batch, off, wt is not None)
    return host_tabs, ind, off, wt, go, counts


def sample_bytes(counts, res, rows_of_tables):
    toff = res.table_offsets
    uniq = [int(toff[i + 1] - toff[i]) for i in range(len(toff) - 1)]
    return metrics.forward_bytes(counts)["total"] + metrics.backward_bytes(counts, uniq)["total"]


def workload_of(args) -> wl.Workload:
    w = wl.get_workload(args.workload)
    if args.tables is not None and args.tables < w.num_tables:
        w = wl.scaled(w, num_tables=args.tables, name=f"{w.name}-first{args.tables}")
    if getattr(args, "rows", None):
        w = wl.scaled(w, rows=args.rows, name=f"{w.name}-rows{args.rows}")
    return w


def cpu_threads() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


# ----------------------------------------------------------------------------- GPU arm

def quantile(xs, q: float) -> float:
    """Linear-interpolated quantile of a non-empty sample."""
    s = sorted(xs)
    k = (len(s) - 1) * q
    lo, hi = math.floor(k), math.ceil(k)
    return s[lo] + (s[hi] - s[lo]) * (k - lo)


def timing_summary(ms):
    return {"median": round(statistics.median(ms), 4), "p10": round(quantile(ms, 0.1), 4),
            "p90": round(quantile(ms, 0.9), 4), "mean": round(statistics.mean(ms), 4),
            "samples": len(ms)}


def run_ours(args):
    from paper_2609_30656_gb300 import tbe

    world, rank, local = dist_env()
    if world > 1:
        torch.distributed.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = workload_of(args)
    seed = args.seed
    tables = wl.make_tables(w, seed, dev)
    batches = [wl.make_batch(w, seed + 1000 * rank, dev, batch_index=k) for k in range(args.rotate)]
    grads_out = [wl.make_grad_out(w, seed + 1000 * rank, dev, batch_index=k)
                 for k in range(args.rotate)]
    # The headline handle records no per-component events: the timed steps carry
    # nothing but the kernels. The breakdown below uses a second handle.
    m = tbe.TBE(tables, pooling="mean" if w.mean else "sum")
    max_n = max(b.num_indices for b in batches)
    m.reserve(w.batch, max_n)
    out = torch.empty(w.batch, w.sum_dims, dtype=torch.float32, device=dev)
    # Size the sparse gradient from a counting pass over every rotating batch.
    U_max, F_max, uniq_tables = 0, 0, []
    for b, go in zip(batches, grads_out):
        probe = m.alloc_grad(0, 0, size_only=True)
        m.backward_into(probe, b.indices, b.offsets, go, b.weights)
        U_max = max(U_max, probe.num_unique)
        F_max = max(F_max, probe.num_floats)
        toff = probe.table_offsets.cpu().tolist()
        uniq_tables.append([toff[t + 1] - toff[t] for t in range(w.num_tables)])
    g = m.alloc_grad(U_max, F_max)
    counts = [metrics.batch_counts(w.dims, w.elem_bytes, w.batch, b.offsets, b.weights is not None)
              for b in batches]
    packed = w.weighted or w.mean
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush = torch.empty(2 * l2, dtype=torch.uint8, device=dev)

    def step(k):
        b, go = batches[k % args.rotate], grads_out[k % args.rotate]
        m.forward(b.indices, b.offsets, b.weights, out=out)
        m.backward_into(g, b.indices, b.offsets, go, b.weights)

    for k in range(args.warmup):
        step(k)
    if m.get_error() != 0:
        raise RuntimeError("device-side error during warm-up")
    torch.cuda.synchronize()

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    stops = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    launches0 = m.launch_count()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        wall0 = time.perf_counter()
        for k in range(args.steps):
            flush.zero_()  # L2 starts cold each step (outside the step's events)
            starts[k].record()
            step(args.warmup + k)
            stops[k].record()
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
    if world > 1:
        torch.distributed.barrier()
    launches = m.launch_count() - launches0
    if m.get_error() != 0:
        raise RuntimeError("device-side error during the timed steps")
    step_ms = [a.elapsed_time(b) for a, b in zip(starts, stops)]
    ms = statistics.median(step_ms)

    # Work of the timed steps (host-side sizes).
    fwd_b, bwd_b, rows_g = 0.0, 0.0, 0.0
    uniq_fwd = 0.0
    for k in range(args.steps):
        i = (args.warmup + k) % args.rotate
        c = counts[i]
        fwd_b += metrics.forward_bytes(c)["total"]
        bwd_b += metrics.backward_bytes(c, uniq_tables[i])["total"]
        uniq_fwd += metrics.forward_unique_bytes(c, uniq_tables[i])
        rows_g += 2 * c.n
    per_step_bytes = (fwd_b + bwd_b) / args.steps
    tot_ms, tot_bytes, tot_rows = aggregate(ms, per_step_bytes, rows_g / args.steps, world)
    gbs = tot_bytes / (tot_ms * 1e-3) / 1e9
    peak, peak_kind = measured_hbm_peak()

    # Per-component breakdown: a separate run with CB_TIMING events between the
    # components, so the headline above carries no event overhead.
    comp_ms, comp_bytes, comp_compulsory = run_breakdown(args, w, tables, batches, grads_out, g, out,
                                                         flush, counts, uniq_tables, packed)
    names = tbe.component_names()
    fwd_ms = sum(comp_ms[n] for n in names if n.startswith("fwd.") and n in comp_ms)
    bwd_ms = sum(comp_ms[n] for n in names if n.startswith("bwd.") and n in comp_ms)
    components = {}
    for n in names:
        if n not in comp_ms:
            continue
        entry = {"ms": round(comp_ms[n], 4), "share": round(comp_ms[n] / (fwd_ms + bwd_ms), 4)}
        if comp_bytes.get(n):
            entry["alg_gbs"] = round(comp_bytes[n] / (comp_ms[n] * 1e-3) / 1e9, 1)
        components[n] = entry
    ceiling = None if args.no_l2 else run_l2_ceiling(dev)
    roofline = roofline_of(w.name, comp_ms, comp_bytes, comp_compulsory, peak, peak_kind, ceiling,
                           counts, w)
    if ceiling and "fwd.gather" in components:
        components["fwd.gather"].update(gather_vs_l2(comp_ms["fwd.gather"], counts, w, ceiling))
    mean_counts_n = statistics.mean(c.n for c in counts)
    fwd_bytes_step = fwd_b / args.steps
    bwd_bytes_step = bwd_b / args.steps
    line = {
        "metric": METRIC, "value": round(gbs, 1), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(tot_ms, 4),
        "step_ms": timing_summary(step_ms),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "storage_dtype": w.dtype, "data": "synthetic",
        "config": {"workload": describe(w),
                   "l2": f"flushed before every step ({2 * l2 >> 20} MB write, outside the "
                         "step's events); inputs also exceed L2",
                   "rotating_batches": args.rotate, "seed": seed,
                   "lookups_per_step": int(mean_counts_n), "parallelism": f"replicas x{world}",
                   "timing": "value and ms_per_step: the median of the per-step CUDA-event times "
                             "(p10/p90 in step_ms) on a handle without component events; "
                             "components: a separate run with CB_TIMING events"},
        "pct_hbm": round(gbs / world / peak, 4), "pct_hbm_nominal": round(gbs / world / NOMINAL_HBM_GBS, 4),
        "rows_per_s": round(tot_rows / (tot_ms * 1e-3), 1),
        "fwd": {"ms": round(fwd_ms, 4), "alg_gbs": round(fwd_bytes_step / (fwd_ms * 1e-3) / 1e9, 1),
                "pct_hbm": round(fwd_bytes_step / (fwd_ms * 1e-3) / 1e9 / peak, 4),
                "rows_per_s": round(mean_counts_n / (fwd_ms * 1e-3), 1),
                "unique_row_gbs": round(uniq_fwd / args.steps / (fwd_ms * 1e-3) / 1e9, 1)},
        "bwd": {"ms": round(bwd_ms, 4), "alg_gbs": round(bwd_bytes_step / (bwd_ms * 1e-3) / 1e9, 1),
                "pct_hbm": round(bwd_bytes_step / (bwd_ms * 1e-3) / 1e9 / peak, 4),
                "rows_per_s": round(mean_counts_n / (bwd_ms * 1e-3), 1)},
        "components": components,
        "roofline": roofline,
        "gpu_launches": int(launches),
        "wall_ms_per_step": round(wall * 1e3 / args.steps, 3),
        "clocks": clk.summary(),
    }
    if ceiling:
        line["l2_ceiling"] = ceiling

    # Next rows: the FM cross term and its gradient on the same pooled output,
    # and the gradient of the per-sample weights on the first batch.
    if not args.no_next:
        nxt = {}
        if len(set(w.dims)) == 1:
            nxt["fm"] = run_fm(w, out, flush, dev, peak)
        nxt["weight_grad"] = run_weight_grad(m, batches[0], grads_out[0], counts[0], flush, peak)
        if all(d % 8 == 0 for d in w.dims):
            nxt["mixed_precision_bf16"] = run_mixed_precision(w, tables, batches[0], grads_out[0], counts[0],
                                                              uniq_tables[0], flush, peak)
        # last: it writes the tables
        nxt["backward_apply"] = run_backward_apply(m, w, batches[0], grads_out[0], counts[0],
                                                   uniq_tables[0], flush, peak, dev, g)
        line["next_rows"] = nxt
    # Component report (Component Benchmark's result table) of this run.
    if args.report and rank == 0:
        write_report(args.report, w, line, comp_ms, comp_bytes, counts, uniq_tables, peak)
    # End to end through the public API from pinned host memory.
    if not args.no_e2e:
        line["e2e"] = run_e2e(args, m, w, batches, grads_out, g, out, dev, world)
    # The oracle on the host cores, rank 0 only, single GPU runs only.
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = run_cpu_baseline(args, w, tables, batches[0], grads_out[0])
    # The reuse-free control: the whole step over uniform indices on the same
    # tables (last: it needs room for ~1.7e8 gradient rows).
    if w.zipf_alpha is not None and not args.no_control:
        go0 = grads_out[0]
        b = go = probe = None
        del g, out, batches, grads_out, b, go, probe
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        line["control_uniform"] = run_control(args, m, w, dev, flush, peak, go0, tables)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def run_breakdown(args, w, tables, batches, grads_out, g, out, flush, counts, uniq_tables, packed,
                  steps=None):
    """Median per-component times (CB_TIMING events between the components) over a
    few steps on a second handle, with their algorithmic and compulsory bytes."""
    from paper_2609_30656_gb300 import tbe
    mt = tbe.TBE(tables, pooling="mean" if w.mean else "sum", timing=True)
    steps = steps or args.breakdown_steps
    rot = len(batches)
    comp = {}
    comp_bytes, comp_compulsory = {}, {}
    for k in range(2 + steps):
        i = k % rot
        b, go = batches[i], grads_out[i]
        flush.zero_()
        mt.forward(b.indices, b.offsets, b.weights, out=out)
        fwd_t = mt.last_timings()
        mt.backward_into(g, b.indices, b.offsets, go, b.weights)
        t = mt.last_timings()
        if k < 2:
            continue
        for n_, v in t.items():
            v = fwd_t[n_] if n_.startswith("fwd.") else v
            if v >= 0:
                comp.setdefault(n_, []).append(v)
        cb = metrics.component_bytes(counts[i], uniq_tables[i], w.rows, packed)
        cc = metrics.component_compulsory_bytes(counts[i], uniq_tables[i], packed)
        for n_, v in cb.items():
            comp_bytes[n_] = comp_bytes.get(n_, 0.0) + v / steps
        for n_, v in cc.items():
            comp_compulsory[n_] = comp_compulsory.get(n_, 0.0) + v / steps
    if mt.get_error() != 0:
        raise RuntimeError("device-side error in the component breakdown")
    mt.close()
    return ({n_: statistics.median(v) for n_, v in comp.items()}, comp_bytes, comp_compulsory)


def roofline_of(workload, comp_ms, comp_bytes, comp_compulsory, peak, peak_kind, ceiling, counts, w):
    """The roofline object of the dominant kernel: the fraction of the HBM copy
    bandwidth its DRAM traffic reaches (ncu bytes per launch, when recorded for
    the current sources, else its compulsory bytes), with the algorithmic and
    L2-gather figures beside it under their own names."""
    dominant = max((n for n in comp_bytes if n in comp_ms), key=lambda n: comp_ms[n])
    t = comp_ms[dominant] * 1e-3
    alg = comp_bytes[dominant]
    comp = comp_compulsory.get(dominant)
    traffic = recorded_traffic(dominant, workload)
    if traffic:
        achieved, basis = traffic / t / 1e9, "dram"
    elif comp:
        achieved, basis = comp / t / 1e9, "compulsory"
    else:  # a streaming kernel without reuse: its algorithmic bytes are compulsory
        achieved, basis = alg / t / 1e9, "algorithmic"
    r = {"bound": "hbm", "kernel": dominant, "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
         "frac": round(achieved / peak, 4), "basis": basis,
         "peak_source": f"{peak_kind} (MEASURED_PEAKS.json hbm_gbs)" if peak_kind == "measured"
         else "fallback 6800 GB/s",
         "traffic": traffic, "launch_ms": round(comp_ms[dominant], 4),
         "compulsory_bytes_per_launch": int(comp) if comp else None,
         "compulsory_frac": round(comp / t / 1e9 / peak, 4) if comp else None,
         "alg_bytes_per_launch": int(alg), "alg_gbs": round(alg / t / 1e9, 1),
         "alg_frac": round(alg / t / 1e9 / peak, 4),
         "note": "achieved/frac: DRAM bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum, "
                 "when recorded for the current sources; else the compulsory bytes: every distinct "
                 "row or grad_out slice once) over the launch's event time; alg_*: every lookup's "
                 "row counted, which exceeds HBM bandwidth when L2 serves the repeats"}
    if ceiling:
        # The gathered part of the kernel against the L2 random-gather rate
        # of rows of the same size.
        if dominant == "bwd.reduce":
            gathered = sum(metrics.backward_bytes(c, [0] * c.num_tables)["grad_gather"] for c in counts) / len(counts)
            row = 4 * max(w.dims)
        else:
            gathered = sum(metrics.forward_bytes(c)["rows"] for c in counts) / len(counts)
            row = w.elem_bytes * max(w.dims)
        key = str(min(512, row))
        if key in ceiling:
            r["l2_gather_gbs"] = round(gathered / t / 1e9, 1)
            r["frac_l2"] = round(gathered / t / 1e9 / ceiling[key]["gbs"], 4)
            r["l2_ceiling_row_bytes"] = int(key)
    return r


def gather_vs_l2(ms: float, counts, w, ceiling) -> dict:
    """The forward gather's row bytes per second against the L2 random-gather
    rate of rows of its size: plain fp32 sums (`frac_l2`) and, for half-precision
    tables, fp16 rows widened into fp32 sums as the gather does (`frac_l2_widened`)."""
    rows = sum(metrics.forward_bytes(c)["rows"] for c in counts) / len(counts)
    key = str(min(512, w.elem_bytes * max(w.dims)))
    if key not in ceiling:
        return {}
    gbs = rows / (ms * 1e-3) / 1e9
    r = {"l2_gather_gbs": round(gbs, 1), "frac_l2": round(gbs / ceiling[key]["gbs"], 4),
         "l2_ceiling_row_bytes": int(key)}
    if w.dtype == "f16" and "f16_sum_gbs" in ceiling[key]:
        r["frac_l2_widened"] = round(gbs / ceiling[key]["f16_sum_gbs"], 4)
    return r


def run_l2_ceiling(dev, reps: int = 5):
    """cb_gather_ceiling on a 33.5 MB row set (one cfg5 table's grad_out slice,
    [65536, 128] fp32) for 512- and 256-byte rows: 2^25 uniformly random rows
    per launch, the median of `reps` launches after two warm-ups."""
    from paper_2609_30656_gb300 import tbe
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    n = 1 << 25
    res = {}
    for row_bytes in (512, 256):
        R = (65536 * 512) // row_bytes
        rows = torch.randn(R, row_bytes // 4, generator=g, device=dev)
        idx = torch.randint(0, R, (n,), generator=g, device=dev, dtype=torch.int32)
        out = torch.empty((n + 31) // 32, dtype=torch.float32, device=dev)
        for _ in range(2):
            tbe.gather_ceiling(rows, idx, out)
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(reps)]
        for a, b in ev:
            a.record()
            tbe.gather_ceiling(rows, idx, out)
            b.record()
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in ev)
        res[str(row_bytes)] = {"gbs": round(n * row_bytes / (ms * 1e-3) / 1e9, 1), "ms": round(ms, 4),
                               "rows": n, "set_mb": round(R * row_bytes / 1e6, 1)}
        # the same rows fetched by TMA gather4
        err = torch.zeros(1, dtype=torch.int32, device=dev)
        for _ in range(2):
            tbe.gather_ceiling(rows, idx, out, tma=True, error=err)
        torch.cuda.synchronize()
        for a, b in ev:
            a.record()
            tbe.gather_ceiling(rows, idx, out, tma=True, error=err)
            b.record()
        torch.cuda.synchronize()
        if int(err.item()) != 0:
            raise RuntimeError("a bounded wait of the TMA gather probe ran out")
        ms = statistics.median(a.elapsed_time(b) for a, b in ev)
        res[str(row_bytes)]["tma_gbs"] = round(n * row_bytes / (ms * 1e-3) / 1e9, 1)
        res[str(row_bytes)]["tma_ms"] = round(ms, 4)
        # fp16 rows of the same size, widened into fp32 sums as the forward does
        rows16 = torch.randn(R, row_bytes // 2, generator=g, device=dev).to(torch.float16)
        for _ in range(2):
            tbe.gather_ceiling(rows16, idx, out)
        torch.cuda.synchronize()
        for a, b in ev:
            a.record()
            tbe.gather_ceiling(rows16, idx, out)
            b.record()
        torch.cuda.synchronize()
        ms = statistics.median(a.elapsed_time(b) for a, b in ev)
        res[str(row_bytes)]["f16_sum_gbs"] = round(n * row_bytes / (ms * 1e-3) / 1e9, 1)
        res[str(row_bytes)]["f16_sum_ms"] = round(ms, 4)
        del rows, rows16, idx, out
    res["how"] = ("cb_gather_ceiling: one warp per 32 random rows of an L2-resident set, 16 bytes per "
                  "lane, 4 row steps in flight, 8 blocks of 256 threads per SM (the walkers' load shape "
                  "without their bookkeeping, at full occupancy); "
                  "tma_*: cb_gather_ceiling_tma, four rows per TMA gather4, 8 gathers in flight per warp; "
                  "f16_sum_*: cb_gather_ceiling_f16, fp16 rows of the same size widened into fp32 sums "
                  "(the forward's 8 mixed-precision adds per 16 bytes)")
    return res


def run_control(args, m, w, dev, flush, peak, go, tables):
    """The whole step (forward + de-duplicated backward) on uniform indices over
    the same tables: no row reuse, so algorithmic bytes ~ DRAM traffic."""
    from paper_2609_30656_gb300 import tbe
    wu = dataclasses.replace(w, zipf_alpha=None)
    batches = [wl.make_batch(wu, args.seed + 7, dev, batch_index=k) for k in range(2)]
    counts = [metrics.batch_counts(w.dims, w.elem_bytes, w.batch, b.offsets, b.weights is not None)
              for b in batches]
    U_max, F_max, uniq = 0, 0, []
    for b in batches:
        probe = m.alloc_grad(0, 0, size_only=True)
        m.backward_into(probe, b.indices, b.offsets, go, b.weights)
        U_max, F_max = max(U_max, probe.num_unique), max(F_max, probe.num_floats)
        toff = probe.table_offsets.cpu().tolist()
        uniq.append([toff[t + 1] - toff[t] for t in range(w.num_tables)])
    g = m.alloc_grad(U_max, F_max)
    out = torch.empty(w.batch, w.sum_dims, dtype=torch.float32, device=dev)
    for k in range(3):
        b = batches[k % 2]
        m.forward(b.indices, b.offsets, b.weights, out=out)
        m.backward_into(g, b.indices, b.offsets, go, b.weights)
    torch.cuda.synchronize()
    steps = 6
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for k in range(steps):
        b = batches[k % 2]
        flush.zero_()
        ev[k][0].record()
        m.forward(b.indices, b.offsets, b.weights, out=out)
        ev[k][1].record()
        m.backward_into(g, b.indices, b.offsets, go, b.weights)
        ev[k][2].record()
    torch.cuda.synchronize()
    if m.get_error() != 0:
        raise RuntimeError("device-side error in the uniform-index control")
    fwd = statistics.median(e[0].elapsed_time(e[1]) for e in ev)
    bwd = statistics.median(e[1].elapsed_time(e[2]) for e in ev)
    stp = statistics.median(e[0].elapsed_time(e[2]) for e in ev)
    fb = statistics.mean(metrics.forward_bytes(counts[k % 2])["total"] for k in range(steps))
    bb = statistics.mean(metrics.backward_bytes(counts[k % 2], uniq[k % 2])["total"] for k in range(steps))
    comp_ms, comp_bytes, comp_compulsory = run_breakdown(
        args, w, tables, batches, [go, go], g, out, flush, counts, uniq, w.weighted or w.mean, steps=4)
    res = {"workload": describe(wu).replace(f"{w.name}:", "cfg5u (same tables):", 1),
           "step_ms": round(stp, 4), "step_alg_gbs": round((fb + bb) / (stp * 1e-3) / 1e9, 1),
           "step_pct_hbm": round((fb + bb) / (stp * 1e-3) / 1e9 / peak, 4),
           "fwd_ms": round(fwd, 4), "fwd_alg_gbs": round(fb / (fwd * 1e-3) / 1e9, 1),
           "fwd_pct_hbm": round(fb / (fwd * 1e-3) / 1e9 / peak, 4),
           "bwd_ms": round(bwd, 4), "bwd_alg_gbs": round(bb / (bwd * 1e-3) / 1e9, 1),
           "bwd_pct_hbm": round(bb / (bwd * 1e-3) / 1e9 / peak, 4),
           "unique_rows": int(sum(uniq[0])),
           "components": {n: round(v, 4) for n, v in comp_ms.items()}}
    for kern in ("fwd.gather", "bwd.reduce"):
        t = comp_ms[kern] * 1e-3
        e = {"ms": round(comp_ms[kern], 4), "alg_gbs": round(comp_bytes[kern] / t / 1e9, 1),
             "alg_frac": round(comp_bytes[kern] / t / 1e9 / peak, 4)}
        traffic = recorded_traffic(kern, "cfg5u")
        e["traffic"] = traffic
        if traffic:
            e["frac_dram"] = round(traffic / t / 1e9 / peak, 4)
        res[kern] = e
    del batches, g, out
    return res


def run_fm(w, y, flush, dev, peak):
    """FM cross term (cb_fm_forward) and its gradient (cb_fm_backward) on the pooled
    output of the last forward: fields = tables, inputs larger than L2."""
    from paper_2609_30656_gb300 import tbe
    T, D, B = w.num_tables, w.dims[0], w.batch
    g = torch.Generator(device=dev)
    g.manual_seed(11)
    grad_fm = torch.randn(B, generator=g, device=dev)
    fm = torch.empty(B, dtype=torch.float32, device=dev)
    grad_y = torch.empty_like(y)
    res = {}
    for name, backward in (("forward", False), ("backward", True)):
        def call():
            if backward:
                tbe.fm_backward(y, grad_fm, T, out=grad_y)
            else:
                tbe.fm_forward(y, T, out=fm)
        for _ in range(2):
            call()
        torch.cuda.synchronize()
        reps = 5
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for a, b in ev:
            flush.zero_()
            a.record()
            call()
            b.record()
        torch.cuda.synchronize()
        ms = statistics.mean(a.elapsed_time(b) for a, b in ev)
        nbytes = metrics.fm_bytes(B, T, D, backward)
        res[name] = {"ms": round(ms, 4), "alg_gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
                     "frac": round(nbytes / (ms * 1e-3) / 1e9 / peak, 4), "bytes": nbytes}
    res["shape"] = f"{B} samples x {T} fields x dim {D} (fp32 pooled rows)"
    del grad_y
    return res


def run_weight_grad(m, b, go, c, flush, peak):
    """d<grad_out, y>/d w for every lookup (cb_tbe_weight_grad) on one batch."""
    gw = torch.empty(b.num_indices, dtype=torch.float32, device=go.device)
    for _ in range(2):
        m.weight_grad(b.indices, b.offsets, go, out=gw)
    torch.cuda.synchronize()
    reps = 5
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for a, e in ev:
        flush.zero_()
        a.record()
        m.weight_grad(b.indices, b.offsets, go, out=gw)
        e.record()
    torch.cuda.synchronize()
    if m.get_error() != 0:
        raise RuntimeError("device-side error in the weight gradient")
    ms = statistics.mean(a.elapsed_time(e) for a, e in ev)
    nbytes = metrics.weight_grad_bytes(c)
    del gw
    return {"ms": round(ms, 4), "alg_gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
            "frac": round(nbytes / (ms * 1e-3) / 1e9 / peak, 4), "bytes": nbytes,
            "note": "algorithmic bytes count each lookup's row and grad_out slice; "
                    "repeated rows and a table's grad_out slice are largely served by L2"}


def run_mixed_precision(w, tables, b, go, c, uniq, flush, peak):
    """Forward and backward of one batch with the pooled output and grad_out in
    bf16 (a second handle over the same tables, CB_OUT_BF16)."""
    from paper_2609_30656_gb300 import tbe
    m = tbe.TBE(tables, pooling="mean" if w.mean else "sum", out_dtype=torch.bfloat16)
    go16 = go.to(torch.bfloat16)
    out = torch.empty(w.batch, w.sum_dims, dtype=torch.bfloat16, device=go.device)
    probe = m.alloc_grad(0, 0, size_only=True)
    m.backward_into(probe, b.indices, b.offsets, go16, b.weights)
    g = m.alloc_grad(probe.num_unique, probe.num_floats)
    res = {}
    for name in ("forward", "backward"):
        def call():
            if name == "forward":
                m.forward(b.indices, b.offsets, b.weights, out=out)
            else:
                m.backward_into(g, b.indices, b.offsets, go16, b.weights)
        for _ in range(2):
            call()
        torch.cuda.synchronize()
        reps = 5
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for a, e in ev:
            flush.zero_()
            a.record()
            call()
            e.record()
        torch.cuda.synchronize()
        ms = statistics.mean(a.elapsed_time(e) for a, e in ev)
        if name == "forward":
            f = metrics.forward_bytes(c)
            nbytes = f["total"] - f["output"] // 2  # bf16 output
        else:
            bb = metrics.backward_bytes(c, uniq)
            nbytes = bb["total"] - bb["grad_gather"] // 2  # bf16 grad_out slices
        res[name] = {"ms": round(ms, 4), "alg_gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
                     "frac": round(nbytes / (ms * 1e-3) / 1e9 / peak, 4), "bytes": nbytes}
    if m.get_error() != 0:
        raise RuntimeError("device-side error in the mixed-precision run")
    m.close()
    del g, out, go16
    return res


def run_backward_apply(m, w, b, go, c, uniq, flush, peak, dev, g):
    """The optimizer step (SGD / row-wise Adagrad) on one batch, fused into the
    backward (cb_tbe_backward_apply), and as a second pass over the gradient the
    backward wrote into `g` (cb_tbe_backward + cb_tbe_apply_sparse). It updates
    the bench's synthetic tables in place, so it runs after every other
    measurement."""
    state = [torch.zeros(r, dtype=torch.float32, device=dev) for r in w.rows]
    res = {}
    reps = 5

    def timed(calls):
        for _ in range(2):
            for f in calls:
                f()
        torch.cuda.synchronize()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(calls) + 1)] for _ in range(reps)]
        for marks in ev:
            flush.zero_()
            marks[0].record()
            for f, e in zip(calls, marks[1:]):
                f()
                e.record()
        torch.cuda.synchronize()
        if m.get_error() != 0:
            raise RuntimeError("device-side error in the optimizer step")
        return [statistics.mean(mk[0].elapsed_time(mk[i + 1]) for mk in ev) for i in range(len(calls))]

    for kind in ("sgd", "adagrad"):
        st = state if kind == "adagrad" else None
        (ms,) = timed([lambda: m.backward_apply(b.indices, b.offsets, go, b.weights, optimizer=kind, lr=1e-3,
                                                eps=1e-8, state=st)])
        nbytes = metrics.apply_step_bytes(c, uniq, kind == "adagrad")
        res[kind] = {"ms": round(ms, 4), "alg_gbs": round(nbytes / (ms * 1e-3) / 1e9, 1),
                     "frac": round(nbytes / (ms * 1e-3) / 1e9 / peak, 4), "bytes": nbytes}
        bwd_ms, total_ms = timed([lambda: m.backward_into(g, b.indices, b.offsets, go, b.weights),
                                  lambda: m.apply_sparse(g, optimizer=kind, lr=1e-3, eps=1e-8, state=st)])
        ab = metrics.sparse_apply_bytes(c, uniq, kind == "adagrad")
        apply_ms = total_ms - bwd_ms
        res[f"{kind}_two_pass"] = {"ms": round(total_ms, 4), "backward_ms": round(bwd_ms, 4),
                                   "apply_ms": round(apply_ms, 4), "apply_bytes": ab,
                                   "apply_gbs": round(ab / (apply_ms * 1e-3) / 1e9, 1),
                                   "apply_frac": round(ab / (apply_ms * 1e-3) / 1e9 / peak, 4)}
    del state
    return res


def write_report(path, w, line, comp_ms, comp_bytes, counts, uniq_tables, peak):
    """Hierarchical component report (JSON and Markdown) of the measured step."""
    from paper_2609_30656_gb300 import report
    steps = len(counts)
    flops = {}
    for c, u in zip(counts, uniq_tables):
        for k, v in metrics.component_flops(c, u, w.mean).items():
            flops[k] = flops.get(k, 0.0) + v / steps
    per_bytes = dict(comp_bytes)  # per step already (the breakdown run's mean)
    extra = {}
    nxt = line.get("next_rows", {})
    if "fm" in nxt:
        B, T, D = w.batch, w.num_tables, w.dims[0]
        extra["fm.forward"] = (nxt["fm"]["forward"]["ms"], nxt["fm"]["forward"]["bytes"], 3.0 * B * T * D)
        extra["fm.backward"] = (nxt["fm"]["backward"]["ms"], nxt["fm"]["backward"]["bytes"], 2.0 * B * T * D)
    if "weight_grad" in nxt:
        g = nxt["weight_grad"]
        extra["weight_grad"] = (g["ms"], g["bytes"], 2.0 * sum(L * d for L, d in zip(counts[0].lookups_per_table, w.dims)))
    for kind in ("sgd", "adagrad"):
        if kind in nxt.get("backward_apply", {}):
            a = nxt["backward_apply"][kind]
            extra[f"backward_apply.{kind}"] = (a["ms"], a["bytes"], flops.get("bwd.reduce", 0.0))
        if f"{kind}_two_pass" in nxt.get("backward_apply", {}):
            a = nxt["backward_apply"][f"{kind}_two_pass"]
            extra[f"apply_sparse.{kind}"] = (a["apply_ms"], a["apply_bytes"], 0.0)
    table_mb = sum(r * d * w.elem_bytes for r, d in zip(w.rows, w.dims)) / 1e6
    root = report.step_tree(comp_ms, per_bytes, flops, table_mb=table_mb, workspace_mb=0.0,
                            extra=extra or None)
    root.children[0].latency_ms = line["ms_per_step"]  # the step as timed
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            tflops = float(json.load(f)["bf16_tflops"])
    except Exception:
        tflops = 1900.0
    meta = {"workload": line["config"]["workload"],
            "note": "bytes and FLOPs are algorithmic; BW util against the measured HBM copy "
                    "bandwidth, MFU against the measured dense bf16 tensor peak"}
    with open(path + ".json", "w") as f:
        f.write(report.to_json(root, peak, tflops, **meta))
    with open(path + ".md", "w") as f:
        f.write(report.to_markdown(root, peak, tflops, title=f"Component report: {w.name}"))


def run_fm_only(args):
    """The FM cross term alone on y ~ N(0, 0.05^2) of shape [batch, T * D]."""
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    w = workload_of(args)
    if len(set(w.dims)) != 1:
        raise SystemExit("the FM cross term needs tables of one dim")
    g = torch.Generator(device=dev)
    g.manual_seed(args.seed)
    y = torch.randn(w.batch, w.sum_dims, generator=g, device=dev).mul_(0.05)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush = torch.empty(2 * l2, dtype=torch.uint8, device=dev)
    peak, _ = measured_hbm_peak()
    with ClockSampler(0) as clk:
        res = run_fm(w, y, flush, dev, peak)
    ms = res["forward"]["ms"] + res["backward"]["ms"]
    nbytes = res["forward"]["bytes"] + res["backward"]["bytes"]
    print(json.dumps({
        "metric": "FM cross term forward + backward, algorithmic HBM GB/s", "unit": "GB/s",
        "value": round(nbytes / (ms * 1e-3) / 1e9, 1), "ms_per_step": round(ms, 4), "n_gpus": 1,
        "higher_is_better": True, "dtype": "f32", "data": "synthetic",
        "config": {"workload": res["shape"]}, "next_rows": {"fm": res}, "clocks": clk.summary()}),
        flush=True)


def run_e2e(args, m, w, batches, grads_out, g, out, dev, world):
    """Forward + backward of a host batch through the public API, every step
    copying its inputs from pinned host memory and its results back to pinned
    host memory: the pooled output [B, sum D] and the row-sparse gradient (ids,
    offsets, values). The value is the pipelined figure: inputs copied on one
    stream into double-buffered device inputs while the previous step computes,
    results copied back on another stream from double-buffered device outputs
    while the next step computes. Also reported: the same with the results left
    on the device (only their sizes read back), and the binding's own serial
    path (host tensors copied on the compute stream, results read after it)."""
    b, go = batches[0], grads_out[0]
    h_ind = b.indices.cpu().pin_memory()
    h_off = b.offsets.cpu().pin_memory()
    h_w = None if b.weights is None else b.weights.cpu().pin_memory()
    h_go = go.cpu().pin_memory()
    steps = max(2, args.steps if args.e2e_steps is None else min(args.steps, args.e2e_steps))
    bytes_in = (h_ind.numel() * 8 + h_off.numel() * 8 + (0 if h_w is None else h_w.numel() * 4)
                + h_go.numel() * 4)
    # This batch's result sizes (from an untimed call): a caller reads the two
    # device scalars to size its copies; here they are fixed for the batch.
    m.forward(b.indices, b.offsets, b.weights, out=out)
    m.backward_into(g, b.indices, b.offsets, go, b.weights)
    U, F = g.num_unique, g.num_floats
    T = w.num_tables
    h_out = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    h_ids = torch.empty(U, dtype=torch.int64).pin_memory()
    h_goff = torch.empty(U + 1, dtype=torch.int64).pin_memory()
    h_grads = torch.empty(F, dtype=torch.float32).pin_memory()
    h_small = torch.empty(2 + T + 1, dtype=torch.int64).pin_memory()
    bytes_out_full = (h_out.numel() * 4 + h_ids.numel() * 8 + h_goff.numel() * 8 + h_grads.numel() * 4
                      + h_small.numel() * 8)
    bytes_out_sizes = h_small.numel() * 8

    def read_sizes(gg):
        h_small[0:1].copy_(gg.num_unique_dev, non_blocking=True)
        h_small[1:2].copy_(gg.num_floats_dev, non_blocking=True)
        h_small[2:].copy_(gg.table_offsets, non_blocking=True)

    def read_all(gg, yy):
        read_sizes(gg)
        h_out.copy_(yy, non_blocking=True)
        h_ids.copy_(gg.unique_ids[:U], non_blocking=True)
        h_goff.copy_(gg.grad_offsets[:U + 1], non_blocking=True)
        h_grads.copy_(gg.grads[:F], non_blocking=True)

    def serial_step():
        # The user's call with host tensors: the binding copies them to the device.
        m.forward(h_ind, h_off, h_w, out=out)
        m.backward_into(g, h_ind, h_off, h_go, h_w)
        read_all(g, out)

    compute = torch.cuda.current_stream(dev)
    copy_in = torch.cuda.Stream(dev)
    copy_out = torch.cuda.Stream(dev)
    ins = [{"ind": torch.empty_like(h_ind, device=dev), "off": torch.empty_like(h_off, device=dev),
            "w": None if h_w is None else torch.empty_like(h_w, device=dev),
            "go": torch.empty_like(h_go, device=dev)} for _ in range(2)]
    outs = [(g, out), (m.alloc_grad(g.unique_ids.numel(), g.grads.numel()), torch.empty_like(out))]
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]  # the step that read this input slot is done
    computed = [torch.cuda.Event() for _ in range(2)]
    drained = [torch.cuda.Event() for _ in range(2)]   # this output slot's results are on the host

    def stage(slot):
        copy_in.wait_event(consumed[slot])
        with torch.cuda.stream(copy_in):
            d = ins[slot]
            d["ind"].copy_(h_ind, non_blocking=True)
            d["off"].copy_(h_off, non_blocking=True)
            if h_w is not None:
                d["w"].copy_(h_w, non_blocking=True)
            d["go"].copy_(h_go, non_blocking=True)
            copied[slot].record(copy_in)

    def pipelined(n, full):
        for e in consumed + drained:
            e.record(compute)
        stage(0)
        for k in range(n):
            slot = k % 2
            if k + 1 < n:
                stage((k + 1) % 2)  # the next step's inputs, while this step computes
            compute.wait_event(copied[slot])
            compute.wait_event(drained[slot])  # step k - 2's results have left this slot
            d = ins[slot]
            gg, yy = outs[slot]
            m.forward(d["ind"], d["off"], d["w"], out=yy)
            m.backward_into(gg, d["ind"], d["off"], d["go"], d["w"])
            consumed[slot].record(compute)
            computed[slot].record(compute)
            copy_out.wait_event(computed[slot])
            with torch.cuda.stream(copy_out):
                if full:
                    read_all(gg, yy)
                else:
                    read_sizes(gg)
                drained[slot].record(copy_out)

    serial_step()
    pipelined(2, True)
    torch.cuda.synchronize()
    counts = metrics.batch_counts(w.dims, w.elem_bytes, w.batch, b.offsets, b.weights is not None)
    toff = g.table_offsets.cpu().tolist()
    uniq = [toff[t + 1] - toff[t] for t in range(T)]
    step_bytes = metrics.forward_bytes(counts)["total"] + metrics.backward_bytes(counts, uniq)["total"]

    def timed(fn):
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        fn()
        torch.cuda.synchronize()
        return (time.perf_counter() - t0) / steps

    el_serial = timed(lambda: [serial_step() for _ in range(steps)])
    el_full = timed(lambda: pipelined(steps, True))
    el_dev = timed(lambda: pipelined(steps, False))
    tot_ms, tot_bytes, _ = aggregate(el_full * 1e3, step_bytes, 0.0, world)
    dev_ms, _, _ = aggregate(el_dev * 1e3, step_bytes, 0.0, world)
    ser_ms, _, _ = aggregate(el_serial * 1e3, step_bytes, 0.0, world)
    if m.get_error() != 0:
        raise RuntimeError("device-side error in the end-to-end run")
    del ins, outs
    return {"value": round(tot_bytes / (tot_ms * 1e-3) / 1e9, 1), "unit": "GB/s",
            "ms_per_step": round(tot_ms, 3), "steps": steps,
            "h2d_bytes_per_step": int(bytes_in), "d2h_bytes_per_step": int(bytes_out_full),
            "serial_ms_per_step": round(ser_ms, 3),
            "result_on_device": {"value": round(tot_bytes / (dev_ms * 1e-3) / 1e9, 1), "unit": "GB/s",
                                 "ms_per_step": round(dev_ms, 3), "d2h_bytes_per_step": int(bytes_out_sizes)},
            "note": "every step copies its host batch (indices, offsets, weights) and grad_out from "
                    "pinned memory and copies the pooled output and the row-sparse gradient (ids, "
                    "offsets, values, sizes) back to pinned memory; value: inputs and results on two "
                    "copy streams with double-buffered device buffers, overlapping the neighbouring "
                    "steps' compute; result_on_device: the same with only the sizes read back; "
                    "serial_ms_per_step: the binding copying host tensors on the compute stream, "
                    "results read after it"}


def run_cpu_baseline(args, w, tables, batch0, go0, budget_s: float | None = None):
    threads = cpu_threads()
    ntab = min(w.num_tables, args.cpu_tables)
    host_tabs, ind, off, wt, go, counts = sample_problem(w, tables, batch0, go0, ntab)
    el, res = oracle_step(host_tabs, ind, off, wt, go, w.batch, w.mean, threads)
    nbytes = sample_bytes(counts, res, w.rows[:ntab])
    out = {"value": round(nbytes / el / 1e9, 3), "unit": "GB/s", "cores": threads,
           "kind": "oracle",
           "sample": f"forward + backward of tables 0..{ntab - 1} of {w.num_tables} at the full "
                     f"batch ({counts.n:,} lookups, {nbytes / 1e9:.2f} GB algorithmic), "
                     f"{el:.1f} s on {threads} threads (OpenMP over bags; the sort is serial)"}
    if not args.no_one_core:
        out["one_core"] = run_one_core(args, tables[0].device)
    return out


def run_one_core(args, dev):
    """The oracle on one host core over the whole of configs 1-3 (forward only for
    config 1, as it is specified), and on all cores beside it."""
    res = {}
    for name in ("cfg1", "cfg2", "cfg3"):
        w = wl.get_workload(name)
        tables = wl.make_tables(w, args.seed, dev)
        b = wl.make_batch(w, args.seed, dev)
        go = wl.make_grad_out(w, args.seed, dev)
        host_tabs, ind, off, wt, go_h, counts = sample_problem(w, tables, b, go, w.num_tables)
        del tables, b, go
        entry = {"lookups": counts.n}
        for cores in (1, cpu_threads()):
            if name == "cfg1":
                import oracle
                t0 = time.perf_counter()
                oracle.forward(host_tabs, w.batch, ind, off, weights=wt, mean=w.mean, threads=cores)
                el = time.perf_counter() - t0
                nb = metrics.forward_bytes(counts)["total"]
            else:
                el, r = oracle_step(host_tabs, ind, off, wt, go_h, w.batch, w.mean, cores)
                nb = sample_bytes(counts, r, w.rows)
            key = "one_core" if cores == 1 else f"{cores}_cores"
            entry[key] = {"ms": round(el * 1e3, 3), "gbs": round(nb / el / 1e9, 4),
                          "rows_per_s": round(counts.n * (1 if name == "cfg1" else 2) / el, 1)}
        entry["what"] = "forward" if name == "cfg1" else "forward + backward"
        res[name] = entry
    return res


# ----------------------------------------------------------------------------- reference arm

def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return  # rank 0 alone times the oracle
    dev = torch.device("cuda", 0) if torch.cuda.is_available() else torch.device("cpu")
    w = workload_of(args)
    threads = cpu_threads()
    ntab = min(w.num_tables, args.ref_tables)
    tables = wl.make_tables(w, args.seed, dev, only=range(ntab))
    b = wl.make_batch(w, args.seed, dev)
    go = wl.make_grad_out(w, args.seed, dev)
    host_tabs, ind, off, wt, gos, counts = sample_problem(w, tables, b, go, ntab)
    # Shrink the sample (batch rows) so the whole run stays within a few minutes.
    el, res = oracle_step(host_tabs, ind, off, wt, gos, w.batch, w.mean, threads)
    budget = args.ref_budget_s / max(1, args.steps + args.warmup)
    frac = min(1.0, budget / max(el, 1e-6))
    keep_b = max(64, int(w.batch * frac))
    if keep_b < w.batch:
        L = (off[1:] - off[:-1]).view(ntab, w.batch)[:, :keep_b]
        new_off = torch.zeros(ntab * keep_b + 1, dtype=torch.int64)
        new_off[1:] = torch.cumsum(L.reshape(-1), 0)
        keep = torch.cat([torch.arange(int(off[t * w.batch]), int(off[t * w.batch]) + int(L[t].sum()))
                          for t in range(ntab)])
        ind, off = ind[keep], new_off
        wt = None if wt is None else wt[keep]
        gos = gos[:keep_b].contiguous()
        counts = metrics.batch_counts([w.dims[t] for t in range(ntab)], w.elem_bytes, keep_b, off,
                                      wt is not None)
    times, nb = [], 0
    for k in range(args.warmup + args.steps):
        el, res = oracle_step(host_tabs, ind, off, wt, gos, keep_b, w.mean, threads)
        if k >= args.warmup:
            times.append(el)
            nb = sample_bytes(counts, res, w.rows[:ntab])
    ms = statistics.mean(times) * 1e3
    gbs = nb / (ms * 1e-3) / 1e9
    sample = (f"forward + backward of tables 0..{ntab - 1} of {w.num_tables}, first {keep_b} of "
              f"{w.batch} batch rows ({counts.n:,} lookups, {nb / 1e9:.3f} GB algorithmic)")
    line = {"impl": "reference", "metric": METRIC, "value": round(gbs, 4), "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": describe(w), "sample": sample, "parallelism": "host cores"},
            "cpu_baseline": {"value": round(gbs, 4), "unit": "GB/s", "cores": threads,
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(gbs, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="cfg5")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--tables", type=int, default=None,
                    help="first N tables only (a smaller case of the same workload)")
    ap.add_argument("--rows", type=int, default=None,
                    help="cap every table's rows (a smaller case for profiling; same lengths and batch)")
    ap.add_argument("--rotate", type=int, default=4)
    ap.add_argument("--e2e-steps", type=int, default=None,
                    help="steps of the end-to-end timing (default: --steps)")
    ap.add_argument("--cpu-tables", type=int, default=32)
    ap.add_argument("--ref-tables", type=int, default=2)
    ap.add_argument("--ref-budget-s", type=float, default=150.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-control", action="store_true",
                    help="skip the step on uniform indices over the same tables")
    ap.add_argument("--no-l2", action="store_true", help="skip the L2 random-gather ceiling leg")
    ap.add_argument("--no-one-core", action="store_true",
                    help="skip the one-core oracle timing of configs 1-3")
    ap.add_argument("--breakdown-steps", type=int, default=5,
                    help="steps of the per-component breakdown run (CB_TIMING handle)")
    ap.add_argument("--no-next", action="store_true",
                    help="skip the next-row measurements (FM cross term)")
    ap.add_argument("--report", default=None,
                    help="write a hierarchical component report to REPORT.json and REPORT.md")
    ap.add_argument("--fm-only", action="store_true",
                    help="time only the FM cross term and its gradient on a synthetic pooled "
                         "output of the workload's shape (no tables are allocated)")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)  # at least three untimed warm-up steps
    if args.impl == "reference":
        run_reference(args)
    elif args.fm_only:
        run_fm_only(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
