#!/usr/bin/env python
"""Benchmark of the GB300 memory lookup: queries/s and roofline fraction.

One step = one htam_query over a batch of the workload's queries (coarse
scores, group top-k, bucketing, fine scores with fused softmax statistics and
top-k, merge) on a prebuilt memory; for the streaming workload a step is one
round (append, then query).  Prints ONE JSON line on rank 0.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the float64 CPU oracle arm

Multi-GPU (launched by torchrun): every rank holds its own replica of the
memory and answers its own query batches; nothing crosses ranks on the data
path (a barrier and a max-reduction of the timing only), so scaling is weak.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2605_29734_gb300 import workloads  # noqa: E402

METRIC = "memory-lookup queries/sec at 1 GB300 and % of roofline (tensor peak or HBM GB/s)"
UNIT = "queries/s"
DEFAULT_WORKLOAD = "uniform_bf16_4m"   # the largest configuration (4,194,304 entries, 32 GiB of keys)
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12   # SMs x FP32 lanes x FMA x max clock


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(workloads.WORKLOADS))
    ap.add_argument("--impl", default="htam", choices=["htam", "reference"])
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--batches", type=int, default=4, help="distinct resident query batches cycled over")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="target length of the oracle sample")
    ap.add_argument("--shrink", type=int, default=1,
                    help="divide the workload's groups and entries by this factor (same group sizes); "
                         "for small profiling captures only")
    ap.add_argument("--stream-rows", type=int, default=None, choices=[0, 1],
                    help="CUDA-core path: stream rows through shared memory (1, library default) or load "
                         "them directly (0)")
    ap.add_argument("--prefix", type=int, default=0,
                    help="prefix-attended queries (htam_query_prefix) of this many states per query; 0 = plain")
    ap.add_argument("--prefix-lambda", type=float, default=0.5, help="position-weight decay of the prefix")
    ap.add_argument("--edges", type=int, default=0,
                    help="route stage 1 by a transition-edge table (htam_query_edges) with prefixes of this "
                         "many earlier groups; 0 = group keys")
    ap.add_argument("--edge-features", type=int, default=12, help="features per edge (12 in App. B.6)")
    ap.add_argument("--flat", action="store_true",
                    help="flat scan (htam_query_flat): every entry a candidate, no group stage")
    ap.add_argument("--unassigned", type=float, default=0.0,
                    help="streaming workloads: this share of each append's rows comes without a group id (-1) "
                         "and joins the group with the nearest key")
    ap.add_argument("--sample", action="store_true",
                    help="draw the groups from the policy of Eq. 11 (htam_query_sampled / "
                         "htam_query_edges_sampled) instead of ranking them")
    ap.add_argument("--tc-pairs", type=int, default=None, choices=[0, 1],
                    help="tensor-core buckets of several chunks on SM pairs (1) or single SMs (0, library default)")
    ap.add_argument("--pdl", type=int, default=None, choices=[0, 1],
                    help="programmatic dependent launch of the query's kernels (1, library default) or plain "
                         "launches (0)")
    ap.add_argument("--fine-overlap", type=int, default=None, choices=[0, 1],
                    help="CUDA-core and tensor-core fine kernels concurrently (1, library default) or in turn (0)")
    ap.add_argument("--tc-min-bucket", type=int, default=None,
                    help="smallest bucket scored on the tensor cores (library default 2)")
    ap.add_argument("--no-secondary", action="store_true",
                    help="default workload only: skip the secondary (4,096-query, 1M-entry) measurement")
    ap.add_argument("--ref-seconds", type=float, default=120.0,
                    help="reference arm: seconds of oracle work over all warm-up and timed steps")
    return ap.parse_args()


def workload_of(args):
    w = workloads.WORKLOADS[args.workload]
    if args.shrink > 1:
        import dataclasses

        # Groups, entries and queries shrink together, so each selected group
        # keeps about the same number of queries (the same kernel regime).
        w = dataclasses.replace(w, name=f"{w.name}_div{args.shrink}", g=w.g // args.shrink, n=w.n // args.shrink,
                                b=max(1, w.b // args.shrink), k_groups=min(w.k_groups, w.g // args.shrink))
    return w


# ----------------------------------------------------------------- plumbing

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def max_over_ranks(x: float, world: int, device: str = "cuda") -> float:
    if world == 1:
        return x
    import torch.distributed as dist

    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(local_seconds: float, local_queries: int, world: int, device: str = "cuda"):
    """Replicas: every rank answers its own batches; the job's rate is all
    ranks' queries over the slowest rank's time.  Returns (rate, max seconds)."""
    slowest = max_over_ranks(local_seconds, world, device)
    return local_queries * world / slowest, slowest


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return {"hbm_gbs": p["hbm_gbs"], "bf16_tflops": p["bf16_tflops"],
                "bf16_tflops_sustained": p.get("bf16_tflops_sustained"), "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "50",
                 "-i", str(device_index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for name, val in zip(names, f[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def read_probe_gbs(dev, gib: int = 4, reps: int = 5) -> float:
    """Context for the HBM roofline: a read-only stream (torch's max of a
    4 GiB fp32 tensor), which a gather that only reads can exceed the
    measured copy peak by.  Best of `reps`, CUDA events."""
    x = torch.ones((gib << 30) // 4, dtype=torch.float32, device=dev)
    x.amax()
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        x.amax()
        b.record()
        torch.cuda.synchronize()
        best = min(best, a.elapsed_time(b) / 1e3)
    n = x.numel() * 4
    del x
    torch.cuda.empty_cache()
    return n / best / 1e9


def source_sha(*names) -> str:
    h = hashlib.sha256()
    for n in names:
        h.update(open(os.path.join(ROOT, "paper_2605_29734_gb300", "csrc", n), "rb").read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, workload: str):
    """Per-launch DRAM bytes of `kernel` on `workload` from a committed ncu
    summary, if the kernel's source is unchanged since the capture."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m_sha = re.search(r"kernel_source_sha:\s*([0-9a-f]+)", text)
    m_tr = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    m_files = re.search(r"kernel_sources:\s*([\w., ]+)", text)
    if not (m_sha and m_tr and m_files):
        return None
    files = [f.strip() for f in m_files.group(1).split(",") if f.strip()]
    if source_sha(*files) != m_sha.group(1):
        return None
    return float(m_tr.group(1))


# ------------------------------------------------------------- algorithmic work

def cuda_core_kernel(w, stream_rows) -> str:
    """Which CUDA-core fine kernel the library runs for this workload: the
    shared-memory row ring for bf16 rows up to 8 KiB (unless turned off),
    otherwise the direct-load kernel."""
    if w.dtype == "bf16" and w.d <= 4096 and stream_rows != 0:
        return "fine_ring"
    return "fine_simt"


def step_work(w, counts: np.ndarray, group_idx: np.ndarray, tc_min: int, flat: bool = False):
    """Algorithmic bytes / flops of one query batch, from the groups it selected:
    each selected group's entries read once, the queries read once, and
    2*D flops per (query, candidate entry); split between the CUDA-core kernel
    (small buckets) and the tensor-core kernel (buckets of >= tc_min queries,
    the memory's routing threshold)."""
    s = 2 if w.dtype == "bf16" else 4
    B, D, G = group_idx.shape[0], w.d, w.g
    sel = group_idx[group_idx >= 0]
    bucket = np.bincount(sel, minlength=G)                # queries per group
    tc_on = w.dtype == "bf16" and w.k_entries <= 32 and tc_min <= B
    is_tc = (bucket >= tc_min) & tc_on
    touched = bucket > 0
    n_b = np.where(group_idx >= 0, counts[np.clip(group_idx, 0, None)], 0).sum(axis=1)
    work = {}
    for name, mask in (("fine", touched & ~is_tc), ("fine_tc", touched & is_tc)):
        entries_read = float(counts[mask].sum())
        queries_read = float(bucket[mask].sum())          # bucket rows staged per kernel
        work[name] = {"bytes": entries_read * D * s + min(B, queries_read) * D * s,
                      "flops": 2.0 * D * float((bucket[mask] * counts[mask]).sum())}
    # The flat scan has no group stage: no group keys read, no coarse scores,
    # no group outputs.
    coarse_flops = 0.0 if flat else 2.0 * D * B * G
    out_bytes = B * ((0 if flat else w.k_groups * 8) + w.k_entries * 12 + 4)
    step_bytes = float(counts[touched].sum()) * D * s + B * D * s + (0 if flat else G * D * 4) + out_bytes
    return {"kernels": work, "step_bytes": step_bytes,
            "step_flops": 2.0 * D * float(n_b.sum()) + coarse_flops, "mean_candidates": float(n_b.mean())}


# --------------------------------------------------------------------- arms

def make_workload(w, seed, device, rank):
    entries, gid, centres = workloads.make_memory(w, seed=seed, device=device)
    return entries, gid, centres


def oracle_rate(w, entries_np, gid_np, queries_np, target_s, cent=None, counts=None, flat=False, sample=False):
    """Times the oracle (as it stands) on a bounded sample of the queries."""
    import oracle

    threads = oracle.default_threads()
    if cent is None and not flat:
        cent, counts = oracle.centroids(entries_np, gid_np, w.g, threads)

    def call(q):
        if flat:
            oracle.flat(entries_np, q, w.k_entries, nthreads=threads)
        elif sample:
            oracle.query_sampled(entries_np, gid_np, w.g, q, w.k_groups, w.k_entries, 1.0, 0.0, 0, 0,
                                 centroid=cent, counts=counts, nthreads=threads)
        else:
            oracle.query(entries_np, gid_np, w.g, q, w.k_groups, w.k_entries, centroid=cent, counts=counts,
                         nthreads=threads)

    probe = min(threads, queries_np.shape[0])
    t0 = time.perf_counter()
    call(queries_np[:probe])
    t_probe = max(time.perf_counter() - t0, 1e-6)
    # Enough queries for about target_s seconds, cycling through the batches
    # when they hold fewer (at most 64 passes).
    n = int(min(64 * queries_np.shape[0], max(probe, probe * target_s / t_probe)))
    n = max(probe, (n // threads) * threads) if n >= threads else n
    reps = -(-n // queries_np.shape[0])
    qs = np.concatenate([queries_np] * reps)[:n] if reps > 1 else queries_np[:n]
    t0 = time.perf_counter()
    call(qs)
    dt = time.perf_counter() - t0
    return n / dt, n, dt, threads, cent, counts


def run_reference(args, world, rank):
    """The float64 oracle on the host cores, same workload, metric and unit."""
    if rank != 0:
        return
    w = workload_of(args)
    device = "cuda" if torch.cuda.is_available() else "cpu"
    entries, gid, centres = make_workload(w, args.seed, device, rank)
    qs = [workloads.make_queries(w, gid, centres, seed=args.seed, stream=4 + 10 * i) for i in range(args.batches)]
    entries_np, gid_np = workloads.to_numpy(entries), workloads.to_numpy(gid)
    del entries
    q_np = np.concatenate([workloads.to_numpy(q) for q in qs])
    import oracle

    threads = oracle.default_threads()
    cent, counts = (None, None) if args.flat else oracle.centroids(entries_np, gid_np, w.g, threads)
    per_step_target = max(0.5, args.ref_seconds / max(1, args.steps + args.warmup))
    if args.flat:  # one query per host thread per step (each scans every entry)
        n_sample = min(threads, q_np.shape[0])
    else:
        _, n_sample, _, _, _, _ = oracle_rate(w, entries_np, gid_np, q_np, per_step_target, cent, counts)
        if n_sample > q_np.shape[0]:  # the sample cycles through the batches
            q_np = np.concatenate([q_np] * -(-n_sample // q_np.shape[0]))
    times = []
    for i in range(args.warmup + args.steps):
        off = (i * n_sample) % max(1, q_np.shape[0] - n_sample + 1)
        t0 = time.perf_counter()
        if args.flat:
            oracle.flat(entries_np, q_np[off:off + n_sample], w.k_entries, nthreads=threads)
        else:
            oracle.query(entries_np, gid_np, w.g, q_np[off:off + n_sample], w.k_groups, w.k_entries,
                         centroid=cent, counts=counts, nthreads=threads)
        if i >= args.warmup:
            times.append(time.perf_counter() - t0)
    total = sum(times)
    value = n_sample * len(times) / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / len(times),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w.name, "queries_per_step": n_sample, "d": w.d, "groups": w.g, "entries": w.n,
                   "k_groups": w.k_groups, "k_entries": w.k_entries, **({"flat": True} if args.flat else {})},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                         "sample": f"{n_sample} queries of {w.name} per step, float64 brute force"
                                   + (", flat retrieval" if args.flat else ", group keys precomputed")},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def measure(args, world, rank, local, full=True):
    """One workload's timed steps on this rank.  Returns the JSON line's
    fields on rank 0 (None elsewhere).  full=False leaves out the end-to-end
    leg and the CPU baseline (the secondary workload of the default run)."""
    from paper_2605_29734_gb300 import htam

    w = workload_of(args)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    props = torch.cuda.get_device_properties(dev)
    l2_bytes = int(getattr(props, "L2_cache_size", 128 << 20))

    entries, gid, centres = make_workload(w, args.seed, dev, rank)
    # The streaming workload appends once per step (warm-up, timed, end-to-end).
    capacity = w.n + (args.warmup + 3 * args.steps + 60) * w.append_per_round if w.rounds else w.n
    mem = htam.Memory(entries, gid, w.g, capacity=capacity)
    if args.stream_rows is not None:
        mem.set_stream_rows(args.stream_rows)
    if args.tc_min_bucket is not None:
        mem.set_tensor_core_min_bucket(args.tc_min_bucket)
    if args.tc_pairs is not None:
        mem.set_tensor_core_pairs(args.tc_pairs)
    if args.pdl is not None:
        mem.set_programmatic_launch(args.pdl)
    if args.fine_overlap is not None:
        mem.set_fine_overlap(args.fine_overlap)
    tc_min = mem.get_tuning(htam.HTAM_TUNE_TC_MIN_BUCKET)
    if args.no_cpu_baseline and not w.rounds:
        del entries                  # the memory holds its own copy
        torch.cuda.empty_cache()
    q_seed = args.seed + 1000 * rank
    P = args.prefix
    if P > 0:
        # A prefix of P states per query, each drawn by the workload's query
        # generator (the most recent last).
        batches = [workloads.make_queries(w, gid, centres, seed=q_seed, stream=4 + 10 * i, b=w.b * P)
                   .view(w.b, P, w.d).contiguous() for i in range(args.batches)]
    else:
        batches = [workloads.make_queries(w, gid, centres, seed=q_seed, stream=4 + 10 * i)
                   for i in range(args.batches)]

    E = args.edges
    if E > 0:
        # A synthetic transition-edge table (features ~ N(0, 1)), a fixed
        # weight vector, and per batch a prefix of E earlier groups per query
        # drawn uniformly (the most recent last).
        rng = np.random.default_rng(args.seed + 7)
        edge_z = torch.randn(w.g, w.g, args.edge_features, device=dev,
                             generator=torch.Generator(device=dev).manual_seed(args.seed + 7))
        edge_w = rng.standard_normal(args.edge_features).astype(np.float32)
        edge_prefix = [rng.integers(0, w.g, (w.b, E)).astype(np.int32) for _ in range(args.batches)]
    batch_of = {id(q): i for i, q in enumerate(batches)}

    def run_query(q, out=None, m=None):
        m = mem if m is None else m
        if args.flat:
            return m.query_flat(q, w.k_entries, out=out)
        if E > 0:
            return m.query_edges(edge_z, edge_w, edge_prefix[batch_of.get(id(q), 0)], args.prefix_lambda, q,
                                 w.k_groups, w.k_entries, out=out,
                                 sampling=(args.seed, batch_of.get(id(q), 0)) if args.sample else None)
        if args.sample:
            return m.query_sampled(q, w.k_groups, w.k_entries, seed=args.seed, offset=batch_of.get(id(q), 0),
                                   out=out)
        if P > 0:
            return m.query_prefix(q, args.prefix_lambda, w.k_groups, w.k_entries, out=out)
        return m.query(q, w.k_groups, w.k_entries, out=out)

    append_batches = []
    if w.rounds:
        n_rounds = args.warmup + args.steps
        append_batches = [workloads.make_append_batch(w, centres, r, seed=args.seed, device=dev)
                          for r in range(min(n_rounds, w.rounds))]
        if args.unassigned > 0:
            gen = torch.Generator(device=dev).manual_seed(args.seed + 31)
            append_batches = [(e, torch.where(torch.rand(g.shape[0], generator=gen, device=dev) < args.unassigned,
                                              torch.full_like(g, -1), g).contiguous()) for e, g in append_batches]
    out = run_query(batches[0])
    torch.cuda.synchronize()

    # Work per batch (the selected groups decide the bytes).
    counts = mem.group_counts().numpy()
    work = []
    for q in batches:
        o = run_query(q)
        if args.flat:  # every query selects every non-empty group
            gi = np.tile(np.flatnonzero(counts > 0).astype(np.int32), (q.shape[0], 1))
        else:
            gi = o["group_idx"].cpu().numpy()
        wk = step_work(w, counts, gi, tc_min, flat=args.flat)
        if P > 0:  # the prefix is read once, in place of the query
            wk["step_bytes"] += (P - 1) * w.b * w.d * (2 if w.dtype == "bf16" else 4)
        if E > 0:  # stage 1 reads the referenced edge-table rows instead of the group keys
            rows = len(np.unique(edge_prefix[len(work)]))
            wk["step_bytes"] += rows * w.g * args.edge_features * 4 - w.g * w.d * 4
            wk["step_flops"] += 2.0 * args.edge_features * E * w.b * w.g - 2.0 * w.d * w.b * w.g
        work.append(wk)
    # The streaming workload's memory grows by one append per step, so the
    # work of step a (append a, then query batch a) is measured on a second
    # memory that replays the same appends and queries: the timed region is
    # steps warmup .. warmup+steps-1, the per-phase pass the next `steps`.
    # Its bytes include the append's: the new rows read and stored, and the
    # touched groups' keys (fp64 sums read and written, fp32 mean and the
    # bf16 halves written).
    stream_work = None
    if w.rounds:
        mem2 = htam.Memory(entries, gid, w.g, capacity=capacity)
        for setter, val in ((mem2.set_stream_rows, args.stream_rows), (mem2.set_tensor_core_min_bucket,
                            args.tc_min_bucket), (mem2.set_tensor_core_pairs, args.tc_pairs)):
            if val is not None:
                setter(val)
        s_elem = 2 if w.dtype == "bf16" else 4
        stream_work = []
        for a in range(args.warmup + 2 * args.steps):
            e, g = append_batches[a % len(append_batches)]
            mem2.append(e, g)
            o = run_query(batches[a % len(batches)], m=mem2)
            counts_a = mem2.group_counts().numpy()
            wk = step_work(w, counts_a, o["group_idx"].cpu().numpy(), tc_min, flat=args.flat)
            touched = int(torch.unique(g[g >= 0]).numel()) if args.unassigned == 0 else w.g
            wk["step_bytes"] += 2.0 * e.shape[0] * w.d * s_elem + touched * w.d * (8 + 8 + 4 + 2 + 2)
            stream_work.append(wk)
        mem2.close()
        if args.no_cpu_baseline:
            del entries
            torch.cuda.empty_cache()

    flush_l2 = work[0]["step_bytes"] < 4 * l2_bytes
    flush = torch.empty(2 * l2_bytes, dtype=torch.uint8, device=dev) if flush_l2 else None

    def one_step(i):
        if w.rounds:
            e, g = append_batches[i % len(append_batches)]
            mem.append(e, g)
        return run_query(batches[i % len(batches)], out=out)

    for i in range(args.warmup):
        one_step(i)
    torch.cuda.synchronize()
    mem.read_phase_timing()          # reset counters
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    sampler = ClockSampler(local)
    time.sleep(0.05)
    barrier(world)
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        if flush is not None:
            flush.fill_(i & 0xFF)
        starts[i].record(stream)
        one_step(args.warmup + i)
        ends[i].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    wall = time.perf_counter() - wall0
    clocks = sampler.stop()
    launches = sum(v[1] for k, v in mem.read_phase_timing().items() if k != "queries")
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    # Per-phase device times from a second pass of the same steps with CUDA
    # events recorded around every phase on the launching stream, and the two
    # fine kernels run one after the other, so that each kernel's duration is
    # its own (in the timed region they share the SMs).  The events separate
    # the kernels, so this pass is not the timed region; it gives the
    # dominant kernel's duration.
    overlap = mem.get_tuning(htam.HTAM_TUNE_FINE_OVERLAP)
    mem.set_fine_overlap(False)
    mem.set_phase_timing(True)
    for i in range(args.steps):
        if flush is not None:
            flush.fill_(i & 0xFF)
        one_step(args.warmup + args.steps + i)
    torch.cuda.synchronize()
    mem.set_phase_timing(False)
    mem.set_fine_overlap(bool(overlap))
    phases = mem.read_phase_timing()
    value, total_s = whole_job_rate(sum(step_ms) / 1e3, w.b * args.steps, world)

    # Dominant kernel roofline (live CUDA events on the launching stream).
    peaks = load_peaks()
    if stream_work is not None:
        per_batch = stream_work[args.warmup:args.warmup + args.steps]
        phase_batch = stream_work[args.warmup + args.steps:]
    else:
        per_batch = [work[(args.warmup + i) % len(work)] for i in range(args.steps)]
        phase_batch = per_batch
    step_bytes = float(np.mean([x["step_bytes"] for x in per_batch]))
    step_flops = float(np.mean([x["step_flops"] for x in per_batch]))
    # The dominant kernel: the fine kernel (CUDA-core or tensor-core) with the
    # most device time in the timed region.
    phase = max(("fine", "fine_tc"), key=lambda k: phases[k][0])
    kernel = {"fine": cuda_core_kernel(w, args.stream_rows), "fine_tc": "fine_tc"}[phase]
    k_ms, k_launches = phases[phase]
    # The phase's device time per step (one launch per step, two when the
    # tensor-core buckets are split between the SM-pair and one-SM kernels).
    k_s = k_ms / 1e3 / args.steps
    k_bytes = float(np.mean([x["kernels"][phase]["bytes"] for x in phase_batch]))
    k_flops = float(np.mean([x["kernels"][phase]["flops"] for x in phase_batch]))
    if phase == "fine_tc":
        tensor_peak = peaks["bf16_tflops_sustained"] or peaks["bf16_tflops"]
        t_hbm = k_bytes / (peaks["hbm_gbs"] * 1e9)
        t_tc = k_flops / (tensor_peak * 1e12)
        if t_tc > t_hbm:
            roofline = {"kernel": kernel, "bound": "tensor", "achieved": k_flops / k_s / 1e12, "peak": tensor_peak,
                        "unit": "TFLOP/s", "peak_note": "measured sustained bf16"}
        else:
            roofline = {"kernel": kernel, "bound": "hbm", "achieved": k_bytes / k_s / 1e9, "peak": peaks["hbm_gbs"],
                        "unit": "GB/s"}
        roofline["tensor_frac"] = k_flops / k_s / 1e12 / tensor_peak
    else:
        roofline = {"kernel": kernel, "bound": "hbm", "achieved": k_bytes / k_s / 1e9, "peak": peaks["hbm_gbs"],
                    "unit": "GB/s", "alu_frac": k_flops / k_s / 1e12 / FP32_ALU_TFLOPS}
    roofline["frac"] = roofline["achieved"] / roofline["peak"]
    if roofline["bound"] == "hbm" and full:
        probe = read_probe_gbs(dev)
        roofline.update({"read_probe_gbs": probe, "frac_of_read_probe": roofline["achieved"] / probe,
                         "read_probe_note": "context only: torch amax over 4 GiB of fp32, read-only, best of 5"})
    # Profiles are per lookup variant: the variant decides the buckets.
    variant = ("_flat" if args.flat else "_sampled" if args.sample else "_edges" if E > 0 else
               "_prefix" if P > 0 else "_unassigned" if args.unassigned > 0 and w.rounds else "")
    roofline.update({"traffic": profiled_traffic(kernel, w.name + variant), "peak_source": peaks["source"],
                     "algorithmic_bytes_per_launch": k_bytes, "flops_per_launch": k_flops,
                     "mean_launch_ms": k_s * 1e3, "launches_per_step": k_launches / args.steps,
                     "duration_source": "CUDA events around the phase on the launching stream, in a second pass "
                                        "of the same steps right after the timed region",
                     "hbm_frac": k_bytes / k_s / 1e9 / peaks["hbm_gbs"]})
    t_roof = max(step_bytes / (peaks["hbm_gbs"] * 1e9),
                 step_flops / ((peaks["bf16_tflops_sustained"] or peaks["bf16_tflops"]) * 1e12))
    step_s = total_s / args.steps

    if not full:
        mem.close()
        if rank != 0:
            return None
        return {"workload": w.name, "value": value, "unit": UNIT, "ms_per_step": 1e3 * step_s, "dtype": w.dtype,
                "config": {"workload": w.name, "queries_per_step": w.b, "d": w.d, "groups": w.g, "entries": w.n,
                           "k_groups": w.k_groups, "k_entries": w.k_entries, "query_batches": len(batches),
                           "l2": ("flushed between steps (2x L2 buffer write, outside the step events)"
                                  if flush_l2 else
                                  f"inputs larger than L2 ({work[0]['step_bytes'] / 1e9:.2f} GB touched per step)")},
                "steps": args.steps, "warmup": args.warmup, "roofline": roofline,
                "step_roofline": {"algorithmic_bytes": step_bytes, "algorithmic_flops": step_flops,
                                  "t_roof_ms": 1e3 * t_roof, "frac": t_roof / step_s,
                                  "phase_ms_per_step": {k: v[0] / args.steps for k, v in phases.items()
                                                        if k != "queries"}},
                "clocks": clocks, "gpu_launches": launches, "wall_s_timed_region": wall}

    # End to end: host (pinned) queries in, host results out, through the C ABI.
    host_q = [b.cpu().pin_memory() for b in batches]
    e2e_steps = max(3, min(args.steps, 50))
    s_elem = 2 if w.dtype == "bf16" else 4
    if P > 0 or E > 0 or args.flat or args.sample:
        # No host-buffer entry point for these lookups: pinned copies on the
        # stream around the call, outputs read back every step.
        dev_q = torch.empty_like(batches[0])
        batch_of[id(dev_q)] = 0
        host_out = {k: torch.empty(v.shape, dtype=v.dtype, pin_memory=True) for k, v in out.items()}

        def e2e_query(i):
            dev_q.copy_(host_q[i % len(host_q)], non_blocking=True)
            batch_of[id(dev_q)] = i % len(host_q)
            o = run_query(dev_q, out=out)
            for k in host_out:
                host_out[k].copy_(o[k], non_blocking=True)
            torch.cuda.current_stream().synchronize()
        entry = ("htam_query_flat" if args.flat else "htam_query_edges" + ("_sampled" if args.sample else "")
                 if E > 0 else "htam_query_sampled" if args.sample else "htam_query_prefix")
        path = f"pinned host queries copied in, {entry}, outputs copied out (torch copies on the stream)"
    else:
        host_out = mem.query_host(host_q[0], w.k_groups, w.k_entries)

        def e2e_query(i):
            mem.query_host(host_q[i % len(host_q)], w.k_groups, w.k_entries, out=host_out)
        path = "htam_query_host (pinned host buffers, copies inside the call)"
    torch.cuda.synchronize()
    barrier(world)
    t0 = time.perf_counter()
    for i in range(e2e_steps):
        if w.rounds:
            e, g = append_batches[i % len(append_batches)]
            mem.append(e, g)
        e2e_query(i)
    barrier(world)
    e2e_s = max_over_ranks(time.perf_counter() - t0, world)
    e2e = {"value": w.b * e2e_steps * world / e2e_s, "unit": UNIT,
           "h2d_bytes_per_step": w.b * max(P, 1) * w.d * s_elem,
           "d2h_bytes_per_step": sum(v.numel() * v.element_size() for v in out.values()), "steps": e2e_steps,
           "path": path}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle

        entries_np, gid_np = workloads.to_numpy(entries), workloads.to_numpy(gid)
        q_np = np.concatenate([workloads.to_numpy(q) for q in batches])
        note = ""
        if P > 0:  # the oracle's prefix reduction (cheap next to the lookup) happens before the timing
            q_np = oracle.round_query(oracle.prefix_reduce(q_np, args.prefix_lambda), w.dtype)
            note = f", prefixes of {P} reduced before timing"
        if args.flat:  # the oracle's flat retrieval on one query per host thread
            threads = oracle.default_threads()
            n = min(w.b, threads)
            t0 = time.perf_counter()
            oracle.flat(entries_np, q_np[:n], w.k_entries, nthreads=threads)
            dt = time.perf_counter() - t0
            rate = n / dt
            note = ", flat retrieval over all entries"
        elif E > 0:  # the oracle's edge-routed lookup on a bounded sample of batch 0
            threads = oracle.default_threads()
            z_np, pre_np = edge_z.cpu().numpy(), edge_prefix[0]
            t0 = time.perf_counter()
            oracle.query_edges(entries_np, gid_np, w.g, z_np, edge_w, pre_np[:threads], args.prefix_lambda,
                               q_np[:threads], w.k_groups, w.k_entries, nthreads=threads)
            t_probe = max(time.perf_counter() - t0, 1e-6)
            n = int(min(w.b, max(threads, threads * args.cpu_seconds / t_probe)))
            t0 = time.perf_counter()
            oracle.query_edges(entries_np, gid_np, w.g, z_np, edge_w, pre_np[:n], args.prefix_lambda, q_np[:n],
                               w.k_groups, w.k_entries, nthreads=threads)
            dt = time.perf_counter() - t0
            rate = n / dt
            note = ", edge-routed (float64 edge scores over the same table)"
        else:
            rate, n, dt, threads, _, _ = oracle_rate(w, entries_np, gid_np, q_np, args.cpu_seconds,
                                                     sample=args.sample)
            if args.sample:
                note += ", groups drawn from the policy"
        cpu = {"value": rate, "unit": UNIT, "cores": threads, "kind": "oracle",
               "sample": f"{n} queries of {w.name} ({dt:.1f} s), float64 brute force over the same memory"
                         + ("" if args.flat else ", group keys precomputed") + note}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1e3 * step_s, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
            "config": {"workload": w.name, "queries_per_step": w.b, "d": w.d, "groups": w.g, "entries": w.n,
                       "k_groups": w.k_groups, "k_entries": w.k_entries, "query_batches": len(batches),
                       "mean_candidates_per_query": float(np.mean([x["mean_candidates"] for x in work])),
                       **({"flat": True} if args.flat else {}),
                       **({"sampled_groups": True} if args.sample else {}),
                       **({"unassigned_share": args.unassigned} if args.unassigned > 0 and w.rounds else {}),
                       "l2": ("flushed between steps (2x L2 buffer write, outside the step events)" if flush_l2 else
                              f"inputs larger than L2 ({work[0]['step_bytes'] / 1e9:.2f} GB touched per step)"),
                       "parallelism": f"replicas{world}" if world > 1 else "single GPU",
                       **({"prefix": P, "prefix_lambda": args.prefix_lambda} if P > 0 else {}),
                       **({"edges_prefix": E, "edge_features": args.edge_features,
                           "prefix_lambda": args.prefix_lambda} if E > 0 else {})},
            "roofline": roofline,
            "step_roofline": {"algorithmic_bytes": step_bytes, "algorithmic_flops": step_flops,
                              "t_roof_ms": 1e3 * t_roof, "frac": t_roof / step_s,
                              "phase_ms_per_step": {k: v[0] / args.steps for k, v in phases.items() if k != "queries"},
                              "fine_kernels": {k: {"bytes": float(np.mean([x["kernels"][k]["bytes"] for x in per_batch])),
                                                   "flops": float(np.mean([x["kernels"][k]["flops"] for x in per_batch]))}
                                               for k in ("fine", "fine_tc")}},
            "e2e": e2e,
            "cpu_baseline": cpu,
            "clocks": clocks,
            "gpu_launches": launches,
            "wall_s_timed_region": wall,
        }
    mem.close()
    return line if rank == 0 else None


# The default run also times the contraction-bound workload (4,096 queries
# against 1,048,576 entries, d = 1,024) after the headline one, in the same
# process, and reports it under "secondary".
SECONDARY_WORKLOAD = "zipf_bf16_1m"


def run_htam(args, world, rank, local):
    line = measure(args, world, rank, local)
    plain = not (args.flat or args.sample or args.prefix or args.edges or args.unassigned > 0 or args.shrink > 1)
    if plain and args.workload == DEFAULT_WORKLOAD and not args.no_secondary:
        import copy

        torch.cuda.empty_cache()
        sec_args = copy.copy(args)
        sec_args.workload = SECONDARY_WORKLOAD
        sec = measure(sec_args, world, rank, local, full=False)
        if line is not None:
            line["secondary"] = sec
    if line is not None:
        print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    world, rank, local = dist_setup()
    try:
        if args.impl == "reference":
            run_reference(args, world, rank)
        else:
            run_htam(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist

            dist.destroy_process_group()


if __name__ == "__main__":
    main()
