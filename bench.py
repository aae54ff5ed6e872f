#!/usr/bin/env python3
"""Throughput of the GB300 ExTernD library: ternary components fitted per second.

One step is one complete decomposition (every block, every ALS iteration, the joint scales and the deflation) of
the workload's matrices. The default workload is the largest single matrix of the benchmark set, the 2560 x 9728
Student-t (nu = 5) MLP up-projection, mu = 3 (k = 7680 components), tau = 1.0, block 128, 4 ALS iterations; its
99.6 MB residual is below the 129 MB L2, so L2 is flushed (a 512 MB write) before every step, inside the timed
region. ``--workload decoder36`` runs the whole 36-layer 4B-class decoder conversion (252 matrices, q/k/v/o/gate/
up/down) back to back on one GPU as one step.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl gb300|reference] [--workload NAME]

With N > 1 (torchrun, one rank per GPU) every rank decomposes its own copy of the workload (independent problems,
no collective on the data path): value = all ranks' components / the slowest rank's time ("scaling": "weak").
``--impl reference`` times the CPU oracle (the plain fp64 restatement of the method) on a bounded sample of the
same workload: the first blocks of the same matrix, which by the greedy prefix property are the same work.

``--row safeguard|refine|packed|sequential`` measures an extension instead (one GPU, its own JSON line): the
decomposition with Prop. 2's safeguard, one refinement sweep (§2.4) of the workload's decomposition, the packed
inference product y = B diag(D) (C x) (§2.6) on factors of the workload's shape, or the sequential algorithm
(§2.3, block width 1) beside the block algorithm on the same matrix.
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
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2607_13511_gb300 import workloads as W  # noqa: E402

METRIC = "ternary components fitted/sec per matrix"
UNIT = "components/s"
DEFAULT_WORKLOAD = W.MLP_UP_2560x9728.name
ROOFLINE_KIND = "products"   # the largest HBM streams of the path: both residual products (profiles/)

# A job is the list of matrices one step decomposes: each single-matrix workload, or the 36-layer conversion.
JOBS = {name: [wl] for name, wl in W.WORKLOADS.items()}
JOBS["decoder36"] = list(W.decoder_conversion())

# dram__bytes_read.sum + dram__bytes_write.sum per launch of the profiled kernel, from one ncu capture, valid
# only while the kernel's source is unchanged (sha256 of the file that holds it).
NCU_TRAFFIC: dict = {
    # ncu --cache-control none (L2 kept across launches, as in the timed graph) of four product_tma_kernel launches
    # in one decomposition of this workload: V-step 45.40 + 37.16 and 44.61 + 13.60 MB, U-step 56.64 + 25.68 and
    # 51.04 + 16.25 MB (read + write); part of the 99.6 MB residual is served from L2
    "kind": "products", "file": "product_tma.cu", "sha": "59887d1810844a9e", "workload": "up2560x9728_t5_mu3_tau1_b128",
    "bytes_per_launch": (45.396992e6 + 37.157376e6 + 44.608256e6 + 13.601536e6 + 56.641280e6 + 25.675008e6 +
                         51.037696e6 + 16.249856e6) / 4,
}


def env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        p = json.load(open(path))
        return p.get("hbm_gbs", 6800.0), "measured"
    return 6800.0, "fallback"


def golden_energy(name):
    path = os.path.join(ROOT, "tests", "golden", "oracle_energies.json")
    try:
        return json.load(open(path))[name]["energy"]
    except (OSError, KeyError, ValueError):
        return None


def workload(name) -> W.Workload:
    """The first (for single-matrix workloads, the only) matrix of a job."""
    return JOBS[name][0]


def block_width(wl):
    return max(1, min(wl.block, min(wl.m, wl.n) // 8))


def inner_rank(wl, mu=None):
    return int(math.floor((wl.mu if mu is None else mu) * min(wl.m, wl.n) + 0.5))


def job_components(wls):
    return sum(inner_rank(wl) for wl in wls)


def _matrix(wl):
    return wl.matrix()


def job_matrices(wls):
    """The job's matrices on the host, generated in a spawned process pool when there are many."""
    if len(wls) <= 4:
        return [wl.matrix() for wl in wls]
    import concurrent.futures
    import multiprocessing
    ctx = multiprocessing.get_context("spawn")
    with concurrent.futures.ProcessPoolExecutor(max_workers=min(16, os.cpu_count() or 1), mp_context=ctx) as pool:
        return list(pool.map(_matrix, wls, chunksize=1))


# ----------------------------------------------------------------------------------------------- CPU oracle
def oracle_sample(wl, budget_blocks):
    """Times the CPU oracle on the first `budget_blocks` blocks of the workload (same matrix, same parameters)."""
    from oracle import externd_oracle as O
    A = wl.matrix()
    h = wl.weights()
    b = block_width(wl)
    k_sample = min(inner_rank(wl), budget_blocks * b)
    mu_sample = k_sample / min(wl.m, wl.n)
    t0 = time.perf_counter()
    res = O.decompose(A, mu_sample, wl.tau, wl.block, wl.iters, h)
    dt = time.perf_counter() - t0
    assert res.D.size == k_sample
    return k_sample, dt


def cpu_cores():
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var, "").isdigit():
            return int(os.environ[var])
    return os.cpu_count()


def sample_workload(name):
    """The matrix a bounded CPU sample of the job runs on: for the decoder, its largest projection (gate)."""
    wls = JOBS[name]
    return max(wls, key=lambda wl: wl.m * wl.n * inner_rank(wl)) if len(wls) > 1 else wls[0]


def run_reference(args):
    rank = env_int("RANK", 0)
    if rank != 0:
        return
    wl = sample_workload(args.workload)
    blocks = args.reference_blocks
    for _ in range(args.warmup):
        oracle_sample(wl, blocks)
    comps, secs = 0, 0.0
    for _ in range(args.steps):
        k, dt = oracle_sample(wl, blocks)
        comps += k
        secs += dt
    value = comps / secs
    sample = f"first {blocks} blocks ({comps // args.steps} of {inner_rank(wl)} components) of {wl.name} per step"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(args.workload),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def config_of(name):
    wls = JOBS[name]
    l2 = "flushed before every step (512 MB write, inside the timed region)"
    if len(wls) == 1:
        wl = wls[0]
        return {"workload": wl.name, "m": wl.m, "n": wl.n, "mu": wl.mu, "k": inner_rank(wl), "tau": wl.tau,
                "block": block_width(wl), "iters": wl.iters, "weighted": wl.weighted, "matrix": wl.kind,
                "seed": wl.seed, "l2": l2}
    shapes = {}
    for wl in wls:
        shapes.setdefault(wl.name.split(".", 1)[1], [wl.m, wl.n, inner_rank(wl)])
    first = wls[0]
    return {"workload": name, "matrices": len(wls), "layers": len({wl.name.split(".")[0] for wl in wls}),
            "shapes_m_n_k": shapes, "k_total": job_components(wls), "mu": first.mu, "tau": first.tau,
            "block": first.block, "iters": first.iters, "weighted": False, "matrix": first.kind,
            "seed": "1000 + 10 * layer + projection index", "l2": l2 + "; 14.5 GB of inputs per step"}


# ----------------------------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.proc = None
        out_dir = os.environ.get("EXTERND_CLOCKS_DIR", tempfile.gettempdir())   # where the raw samples go
        self.path = os.path.join(out_dir, f"clocks_rank{env_int('RANK', 0)}.csv")
        self.idx = device_index

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, ValueError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.25)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return None
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


# ----------------------------------------------------------------------------------------------- GPU arm
def algorithmic_bytes(kind, wl):
    """Bytes one launch of the kernel class must move at minimum (R dominates; ternary factors are int8)."""
    m, n, b = wl.m, wl.n, block_width(wl)
    hbytes = 4 * n if wl.weighted else 0
    if kind == "vstep":      # read R and U, write U^T R
        return 4 * m * n + m * b + 4 * b * n
    if kind == "ustep":      # read R, V (and h), write R H V
        return 4 * m * n + n * b + hbytes + 4 * m * b
    if kind == "products":   # V-steps and U-steps launch equally often
        return (algorithmic_bytes("vstep", wl) + algorithmic_bytes("ustep", wl)) / 2
    if kind == "deflate":    # read and write R, read U, V, d
        return 8 * m * n + (m + n) * b + 4 * b + hbytes
    if kind == "sequential":   # the one-launch b = 1 fit: R in shared memory, per component the start's column
        # energies and column, 2 iters products and the deflation's read and write: (2 iters + 3) 4mn bytes
        return inner_rank(wl) * (2 * wl.iters + 3) * 4 * m * n
    raise ValueError(kind)


# Shared-memory roofline of the one-launch sequential kernel: its cluster's 8 SMs, 128 bytes per SM per clock
# (32 banks x 4 bytes) at the 2070 MHz maximum SM clock.
SEQ_SMEM_GBS = 8 * 128 * 2.07


def sequential_workload(wl):
    """Block width 1 and a residual that fits the cluster kernel's shared memory (8 CTAs, <= 200 KB each)."""
    rpc = -(-wl.m // 8)
    return block_width(wl) == 1 and wl.n <= 4096 and (rpc * wl.n + 5 * wl.n + 2 * rpc) * 4 <= 200 * 1024


def decomposition_bytes(wl):
    """Least HBM traffic of one whole decomposition: per block 2 * iters passes over R plus the read-modify-write
    of the deflation, plus the initial copy R = A (read A, write R)."""
    nblocks = -(-inner_rank(wl) // block_width(wl))
    return nblocks * (2 * wl.iters * 4 + 8) * wl.m * wl.n + 8 * wl.m * wl.n


def max_over_ranks(value, device, world):
    """The largest of the ranks' values, returned on every rank (value itself for one rank)."""
    import torch
    import torch.distributed as dist

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, units_per_rank, ms):
    """Whole-job throughput: every rank's units over the slowest rank's time (weak scaling, replicas)."""
    return world * units_per_rank / (ms / 1e3)


def source_sha(path):
    return hashlib.sha256(open(path, "rb").read()).hexdigest()[:16]


def run_gpu(args):
    import torch
    import torch.distributed as dist

    rank, world, local = env_int("RANK", 0), env_int("WORLD_SIZE", 1), env_int("LOCAL_RANK", 0)
    wls = JOBS[args.workload]
    host_A = job_matrices(wls)          # before the first CUDA call (the pool is spawned, not forked)

    import paper_2607_13511_gb300 as X

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    X.load()

    host_A = [torch.from_numpy(a) for a in host_A]
    host_h = [None if wl.weights() is None else torch.from_numpy(wl.weights()) for wl in wls]
    As = [a.to(dev) for a in host_A]
    hs = [None if h is None else h.to(dev) for h in host_h]
    ks = [X.rank(wl.m, wl.n, wl.mu) for wl in wls]
    outs = [(torch.empty((wl.m, k), dtype=torch.int8, device=dev), torch.empty((k,), dtype=torch.float32, device=dev),
             torch.empty((k, wl.n), dtype=torch.int8, device=dev)) for wl, k in zip(wls, ks)]
    flush = torch.empty(128 * 1024 * 1024, dtype=torch.float32, device=dev)   # 512 MB > L2
    comps = sum(ks)

    def step():
        energies, launches = [], 0
        for i, wl in enumerate(wls):
            energies.append(X.decompose(As[i], wl.mu, wl.tau, wl.block, wl.iters, hs[i], out=outs[i]).energy)
            launches += X.kernel_launches()
        return energies, launches

    for _ in range(args.warmup):
        flush.fill_(0.0)
        step()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    # ---- timed region: K steps, device-timed with CUDA events on the current stream
    stream = torch.cuda.current_stream(dev)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    launches = 0
    with ClockSampler(local) as clocks:
        barrier()
        ev0.record(stream)
        for i in range(args.steps):
            flush.fill_(float(i))
            energies, nl = step()
            launches += nl
        ev1.record(stream)
        barrier()
    ms_max = max_over_ranks(ev0.elapsed_time(ev1), dev, world)
    value = job_rate(world, comps * args.steps, ms_max)

    if args.steps_only:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
                              "warmup": args.warmup, "ms_per_step": ms_max / args.steps, "gpu_launches": launches,
                              "config": config_of(args.workload), "steps_only": True}), flush=True)
        if world > 1:
            dist.destroy_process_group()
        return

    # ---- end to end through the host entry point: H2D of A (and h), decomposition, D2H of B, D, C, energy
    A_pin = [a.pin_memory() for a in host_A]
    h_pin = [None if h is None else h.pin_memory() for h in host_h]
    hout = {}
    for wl, k in zip(wls, ks):
        if (wl.m, wl.n, k) not in hout:
            hout[(wl.m, wl.n, k)] = (torch.empty((wl.m, k), dtype=torch.int8, pin_memory=True),
                                     torch.empty((k,), dtype=torch.float32, pin_memory=True),
                                     torch.empty((k, wl.n), dtype=torch.int8, pin_memory=True))

    def e2e_step():
        for i, (wl, k) in enumerate(zip(wls, ks)):
            X.decompose_host(A_pin[i], wl.mu, wl.tau, wl.block, wl.iters, h_pin[i], out=hout[(wl.m, wl.n, k)])

    for _ in range(max(1, min(args.warmup, 2))):
        e2e_step()
    barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.steps):
        flush.fill_(float(i))
        e2e_step()
    e1.record(stream)
    barrier()
    e2e_value = job_rate(world, comps * args.steps, max_over_ranks(e0.elapsed_time(e1), dev, world))
    h2d = sum(4 * wl.m * wl.n + (4 * wl.n if wl.weighted else 0) for wl in wls)
    d2h = sum(wl.m * k + k * wl.n + 4 * k + 8 for wl, k in zip(wls, ks))

    # ---- live roofline of the dominant kernel class: event pairs inside the graph, over a second timed pass
    kind = args.roofline_kind
    seq = all(sequential_workload(wl) for wl in wls)
    if seq:   # the whole fit is one kernel (profiled as the solve class)
        kind = "sequential"
    X.profile("solve" if seq else kind)
    for _ in range(2):
        flush.fill_(0.0)
        step()
    prof_ms, prof_n, prof_bytes = 0.0, 0, 0.0
    for i in range(args.steps):
        flush.fill_(float(i))
        for j, wl in enumerate(wls):
            X.decompose(As[j], wl.mu, wl.tau, wl.block, wl.iters, hs[j], out=outs[j])
            a, b = X.profile_read()
            prof_ms += a
            prof_n += b
            prof_bytes += b * algorithmic_bytes(kind, wl)
    X.profile("off")
    per_launch_s = prof_ms / 1e3 / max(prof_n, 1)
    bytes_per_launch = prof_bytes / max(prof_n, 1)
    achieved = bytes_per_launch / per_launch_s / 1e9 if per_launch_s > 0 else 0.0
    peak, peak_src = peaks()
    bound = "hbm"
    if seq:
        bound, peak, peak_src = "smem", SEQ_SMEM_GBS, "derived: 8 SMs x 128 B/clock x 2070 MHz"
    traffic = None
    src = os.path.join(ROOT, "paper_2607_13511_gb300", "csrc", NCU_TRAFFIC.get("file", "gemm.cu"))
    if NCU_TRAFFIC.get("kind") == kind and os.path.exists(src) and NCU_TRAFFIC.get("sha") == source_sha(src) \
            and NCU_TRAFFIC.get("workload") == args.workload:
        traffic = NCU_TRAFFIC["bytes_per_launch"]

    # ---- what this GPU's HBM delivers to a plain read stream (context for the products' fraction, not the peak):
    # torch's float32 sum over 2 GB, best of 5, CUDA events
    rbuf = torch.ones(512 * 1024 * 1024, dtype=torch.float32, device=dev)
    for _ in range(2):
        rbuf.sum()
    best = float("inf")
    for _ in range(5):
        r0, r1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        r0.record(stream)
        rbuf.sum()
        r1.record(stream)
        r1.synchronize()
        best = min(best, r0.elapsed_time(r1))
    read_gbs = rbuf.numel() * 4 / (best / 1e3) / 1e9
    del rbuf

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    step_bytes = sum(decomposition_bytes(wl) for wl in wls)
    ms_step = ms_max / args.steps
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded numpy PCG64; see workloads.py)",
        "config": {**config_of(args.workload), "parallelism": f"replicas x{world}"},
    }
    deltas = {}
    for wl, e in zip(wls, energies):
        g = golden_energy(wl.name)
        if g is not None:
            deltas[wl.name] = e - g
    if len(wls) == 1:
        line["energy"] = energies[0]
        line["delta_E_vs_oracle"] = deltas.get(wls[0].name)
    else:
        line["energy"] = {"min": min(energies), "median": statistics.median(energies), "max": max(energies)}
        line["delta_E_vs_oracle"] = {"matrices": len(deltas),
                                     "max_abs": max((abs(d) for d in deltas.values()), default=None),
                                     "per_matrix": deltas}
    line["e2e"] = {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                   "path": "externd_decompose_host (pinned host buffers)"}
    line["gpu_launches"] = launches
    line["roofline"] = {"bound": bound, "kernel": kind, "achieved": achieved, "peak": peak, "unit": "GB/s",
                        "frac": achieved / peak, "traffic": traffic, "peak_source": peak_src,
                        "bytes_per_launch": bytes_per_launch, "launches": prof_n,
                        "us_per_launch": per_launch_s * 1e6}
    if not seq:
        line["read_ceiling"] = {"gbs": read_gbs, "frac_of_peak": read_gbs / peak,
                                "roofline_frac_of_it": achieved / read_gbs,
                                "how": "torch float32 sum over 2 GB on this GPU, best of 5 (a read-only stream)"}
    if not seq:   # the HBM model of the whole step: 2 iters passes over R and the deflation per block
        line["step_roofline"] = {"algorithmic_bytes": step_bytes, "lower_bound_ms": step_bytes / (peak * 1e6),
                                 "frac": step_bytes / (peak * 1e6) / ms_step}
    cs = clocks.summary()
    if cs is not None:
        line["clocks"] = cs
    if world == 1 and not args.no_cpu_baseline:
        swl = sample_workload(args.workload)
        kk, dt = oracle_sample(swl, args.cpu_blocks)
        line["cpu_baseline"] = {"value": kk / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                                "sample": f"first {args.cpu_blocks} blocks ({kk} of {inner_rank(swl)} components) "
                                          f"of {swl.name}, {dt:.1f} s"}
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ----------------------------------------------------------------------------------------------- extension rows
def time_steps(torch, stream, steps, fn, flush=None):
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    ev0.record(stream)
    out = None
    for i in range(steps):
        if flush is not None:
            flush.fill_(float(i))
        out = fn()
    ev1.record(stream)
    torch.cuda.synchronize()
    return ev0.elapsed_time(ev1) / steps, out


def run_row(args):
    """One JSON line for an extension row, on cuda:0."""
    import numpy as np
    import torch

    import paper_2607_13511_gb300 as X
    from oracle import externd_next as N
    from oracle import externd_oracle as O

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    X.load()
    wl = workload(args.workload)
    stream = torch.cuda.current_stream(dev)
    k = X.rank(wl.m, wl.n, wl.mu)
    peak, peak_src = peaks()
    line = {"row": args.row, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "vs_baseline": None,
            "data": "synthetic (seeded numpy PCG64; see workloads.py)", "config": config_of(wl.name)}
    if args.row in ("safeguard", "refine"):
        A_np = wl.matrix()
        A = torch.from_numpy(A_np).to(dev)
        h_np = wl.weights()
        h = None if h_np is None else torch.from_numpy(h_np).to(dev)
        flush = torch.empty(128 * 1024 * 1024, dtype=torch.float32, device=dev)   # 512 MB > L2
        bufs = lambda: (torch.empty((wl.m, k), dtype=torch.int8, device=dev),
                        torch.empty((k,), dtype=torch.float32, device=dev),
                        torch.empty((k, wl.n), dtype=torch.int8, device=dev))
        out_plain, out_ext = bufs(), bufs()
        plain = lambda: X.decompose(A, wl.mu, wl.tau, wl.block, wl.iters, h, out=out_plain)
        for _ in range(args.warmup):
            dec = plain()
        ms_plain, dec = time_steps(torch, stream, args.steps, plain, flush)
        b = block_width(wl)
        if args.row == "safeguard":
            fn = lambda: X.decompose_safeguarded(A, wl.mu, wl.tau, wl.block, wl.iters, h, out=out_ext)
            for _ in range(args.warmup):
                fn()
            ms, (res, act) = time_steps(torch, stream, args.steps, fn, flush)
            kk = min(k, args.cpu_blocks * b)
            t0 = time.perf_counter()
            N.decompose_safeguarded(A_np, kk / min(wl.m, wl.n), wl.tau, wl.block, wl.iters, h_np)
            dt = time.perf_counter() - t0
            line.update({"metric": "ternary components fitted/sec per matrix, Prop. 2 safeguard on", "unit": UNIT,
                         "value": k / (ms / 1e3), "ms_per_step": ms, "higher_is_better": True, "dtype": "f32",
                         "energy": res.energy, "activations": act, "plain_ms_per_step": ms_plain,
                         "overhead_vs_plain": ms / ms_plain - 1.0,
                         "cpu_baseline": {"value": kk / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                                          "sample": f"first {kk} components of {wl.name} with the safeguard, "
                                                    f"{dt:.1f} s"}})
        else:
            fn = lambda: X.refine(A, dec, wl.tau, wl.block, wl.iters, 1, h, out=out_ext)
            for _ in range(args.warmup):
                fn()
            ms, (ref, rep) = time_steps(torch, stream, args.steps, fn, flush)
            # oracle: one sweep over the first blocks' factorization (a prefix of the same run)
            kk = min(k, max(1, args.cpu_blocks // 4) * b)
            res_o = O.decompose(A_np, kk / min(wl.m, wl.n), wl.tau, wl.block, wl.iters, h_np)
            t0 = time.perf_counter()
            N.refine(A_np, res_o, wl.tau, wl.block, wl.iters, 1, h_np)
            dt = time.perf_counter() - t0
            line.update({"metric": "components refitted/sec (one refinement sweep, §2.4)", "unit": UNIT,
                         "value": k / (ms / 1e3), "ms_per_step": ms, "higher_is_better": True, "dtype": "f32",
                         "energy_before": dec.energy, "energy_after": ref.energy, "blocks_replaced": rep[0],
                         "decompose_ms_per_step": ms_plain,
                         "cpu_baseline": {"value": kk / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                                          "sample": f"one sweep over the first {kk} components of {wl.name}, "
                                                    f"{dt:.1f} s"}})
    elif args.row == "sequential":
        # §2.3 against §2.4 on the same matrices: the sequential algorithm (block width 1) and the block algorithm
        # at the cap, the same number of components; the paper reports about 16x for block over sequential (§3.1)
        cases = []
        for wl_s, block, mu in ((W.SEQUENTIAL_256, 32, None), (W.MLP_UP_2560x9728, 128, 256 / 2560)):
            A = torch.from_numpy(wl_s.matrix()).to(dev)
            mu_c = wl_s.mu if mu is None else mu
            kk = X.rank(wl_s.m, wl_s.n, mu_c)
            res = {}
            for b in (1, block):
                fn = lambda b=b: X.decompose(A, mu_c, wl_s.tau, b, wl_s.iters)
                for _ in range(max(1, args.warmup)):
                    fn()
                reps = 3 if (b == 1 and wl_s.m * wl_s.n > 1 << 20) else args.steps
                ms, dec = time_steps(torch, stream, reps, fn)
                res[b] = {"ms": ms, "components_per_s": kk / (ms / 1e3), "energy": dec.energy,
                          "launches": X.kernel_launches()}
            cases.append({"matrix": wl_s.name, "m": wl_s.m, "n": wl_s.n, "k": kk, "tau": wl_s.tau,
                          "iters": wl_s.iters, "sequential_b1": res[1], f"block_b{block}": res[block],
                          "block_over_sequential": res[block]["components_per_s"] / res[1]["components_per_s"]})
        line.update({"metric": "ternary components fitted/sec, sequential (§2.3) and block (§2.4) on the same matrix",
                     "unit": UNIT, "value": cases[0]["sequential_b1"]["components_per_s"],
                     "ms_per_step": cases[0]["sequential_b1"]["ms"], "higher_is_better": True, "dtype": "f32",
                     "cases": cases,
                     "paper_context": "about 16x block over sequential on one AMD MI50 (torch), §3.1 / Table 1"})
    else:   # packed inference product
        m, n = wl.m, wl.n
        layer_bytes = (m * k + k * n) / 4.0                    # 2 bits per ternary entry
        copies = max(2, math.ceil(2 * 129e6 / layer_bytes))   # rotate through more than twice the L2
        g = torch.Generator(device=dev).manual_seed(wl.seed)
        layers = []
        for _ in range(copies):
            Bt = torch.randint(-1, 2, (m, k), dtype=torch.int8, device=dev, generator=g)
            Ct = torch.randint(-1, 2, (k, n), dtype=torch.int8, device=dev, generator=g)
            D = torch.rand(k, device=dev, generator=g) + 0.1
            layers.append((X.pack_ternary(Bt), D, X.pack_ternary(Ct)))
            del Bt, Ct
        x = torch.randn(n, device=dev, generator=g)
        for _ in range(args.warmup):
            for L in layers:
                X.ternary_apply(L[0], L[1], L[2], x)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            for L in layers:
                X.ternary_apply(L[0], L[1], L[2], x)
        graph.replay()
        ms, _ = time_steps(torch, stream, args.steps, graph.replay)
        per_apply = ms / copies
        bytes_apply = layer_bytes + 4 * (n + 2 * k + m)
        achieved = bytes_apply / (per_apply / 1e3) / 1e9
        # oracle: the float64 product on the host, a few applies of one layer
        rng = np.random.default_rng(wl.seed)
        Bn = rng.integers(-1, 2, (m, k)).astype(np.int8)
        Cn = rng.integers(-1, 2, (k, n)).astype(np.int8)
        Dn, xn = rng.random(k) + 0.1, rng.standard_normal(n)
        reps, t0 = 0, time.perf_counter()
        while reps < 3 or time.perf_counter() - t0 < 2.0:
            N.ternary_apply(Bn, Dn, Cn, xn)
            reps += 1
        dt = (time.perf_counter() - t0) / reps
        line.update({"metric": "packed ternary products y = B diag(D) (C x) per second", "unit": "products/s",
                     "value": 1e3 / per_apply, "ms_per_step": ms, "higher_is_better": True, "dtype": "bf16x3 (exact f32 split)",
                     "us_per_product": per_apply * 1e3, "layers_rotated": copies,
                     "roofline": {"bound": "hbm", "kernel": "apply (fragments + 2 packed products)",
                                  "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                                  "traffic": None, "peak_source": peak_src, "bytes_per_launch": bytes_apply},
                     "gpu_launches": 3 * copies * args.steps,
                     "cpu_baseline": {"value": 1.0 / dt, "unit": "products/s", "cores": cpu_cores(),
                                      "kind": "oracle", "sample": f"{reps} float64 products of one {m}x{k}x{n} "
                                                                  f"layer, {dt * reps:.1f} s"}})
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(JOBS))
    ap.add_argument("--roofline-kind", default=ROOFLINE_KIND, choices=["products", "vstep", "ustep", "deflate"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--steps-only", action="store_true",
                    help="time the steps and print the line without the e2e, roofline and CPU passes (profiler runs)")
    ap.add_argument("--cpu-blocks", type=int, default=16, help="blocks of the workload the CPU baseline times")
    ap.add_argument("--reference-blocks", type=int, default=2, help="blocks per step of the reference arm")
    ap.add_argument("--row", default="decompose", choices=["decompose", "safeguard", "refine", "packed", "sequential"],
                    help="an extension row instead of the headline decomposition (one GPU)")
    args = ap.parse_args()
    if args.row != "decompose":
        run_row(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
