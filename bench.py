#!/usr/bin/env python3
"""Benchmark of serially-equivalent sparse SGD on GB300.

One step = the whole hot path over one synthetic problem held in HBM:
pdb_build_conflicts (validate, feature sort, chains) + pdb_schedule_build +
pdb_sgd_epoch over all of the workload's epochs.  The metric is
nnz-updates per second (epochs x nnz / step time).  Default workload: the
low-conflict, HBM-bound problem (4e6 examples x 1e8 features, 100 uniform
ids per example, squared loss, eta = 1e-3, 2 epochs).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun each rank runs an independent replica on its own GPU (the
method's conflict structure does not shard without a per-hop exchange), and
the aggregate is the sum of all ranks' updates over the slowest rank's time.
``--impl reference`` times the CPU oracle (sequential SGD, one core) on a
bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

# The end-to-end measurement runs four streams at once (compute, host-to-device
# copies, device-to-host copies, the library's own stream for frees).  With the
# default 8 hardware work queues per device some of them share a queue, and
# work on one then waits behind a long copy on another; 32 queues keep them
# apart.  Read when the CUDA context is created, so it is set before anything
# imports torch.
os.environ.setdefault("CUDA_DEVICE_MAX_CONNECTIONS", "32")

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "serially-equivalent sparse SGD nnz-updates/sec at 1 GB300; % of HBM roofline"
UNIT = "nnz-updates/s"
ALG_BYTES_PER_NNZ = 16      # col 4 + val 4 + w read 4 + w write 4
ALG_BYTES_PER_ROW = 12      # row_ptr 8 + y 4
L2_BYTES = 129 * 2 ** 20


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="low-conflict")
    ap.add_argument("--mode", choices=["auto", "ready", "levels", "chain", "window"], default="auto")
    ap.add_argument("--rows", type=int, default=None, help="override the workload's example count")
    ap.add_argument("--ticket-chunk", type=int, default=0, help="READY engine: examples per ticket (0 = default)")
    ap.add_argument("--blocks-per-sm", type=int, default=0)
    ap.add_argument("--bsp", type=int, default=0,
                    help="time pdb_bsp_epoch with this mini-batch instead of pdb_sgd_epoch (-1: the workload's own)")
    ap.add_argument("--delay", type=int, default=None,
                    help="time pdb_ssp_epoch (admissible delay, READY schedule) with this delay instead")
    ap.add_argument("--ssp-gates", choices=["count", "prefix"], default="count",
                    help="with --delay: counting gates, or prefix gates (a writer waits for the slowest reader)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="target length of the CPU oracle sample")
    return ap.parse_args(argv)


# ---------------------------------------------------------------- distributed helpers
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def reduce_max(value: float, world: int) -> float:
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def reduce_sum(value: float, world: int) -> float:
    if world == 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------------- measurement helpers
def measured_peak_hbm():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, local_rank: int):
        self.gpu = self.smi_id(local_rank)
        self.proc = None
        self.file = None

    @staticmethod
    def smi_id(local_rank: int) -> str:
        """nvidia-smi id of the CUDA device this process uses (PCI bus id when torch knows it)."""
        try:
            import torch
            props = torch.cuda.get_device_properties(local_rank)
            bus = getattr(props, "pci_bus_id", None)
            dom = getattr(props, "pci_domain_id", None)
            dev = getattr(props, "pci_device_id", None)
            if bus is not None and dom is not None and dev is not None:
                return "%08X:%02X:%02X.0" % (dom, bus, dev)
        except Exception:
            pass
        vis = os.environ.get("CUDA_VISIBLE_DEVICES")
        if vis:
            ids = [x.strip() for x in vis.split(",") if x.strip()]
            if local_rank < len(ids):
                return ids[local_rank]
        return str(local_rank)

    def __enter__(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.file is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "gpu": self.gpu}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1])]
        mx = [num(r[2]) for r in rows if num(r[2])]
        pw = [num(r[3]) for r in rows if num(r[3])]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None, "samples": len(rows), "reasons": reasons, "gpu": self.gpu}


def cpu_baseline(problem, target_s: float):
    """The oracle (sequential SGD, one thread): the whole workload when that
    takes at most ~3x target_s, else the first R examples sized to ~target_s."""
    import oracle
    n = problem.n_rows
    k_mean = problem.nnz / max(n, 1)
    rows = min(n, 200000)
    t0 = time.perf_counter()
    oracle.sgd(problem, epochs=1, rows=rows)
    dt = time.perf_counter() - t0
    per_nnz = dt / max(1, int(problem.row_ptr[rows]))
    if per_nnz * problem.nnz * problem.epochs <= 3 * target_s:
        t0 = time.perf_counter()
        oracle.sgd(problem)
        dt = time.perf_counter() - t0
        nnz = problem.nnz * problem.epochs
        sample = (f"the whole workload: {n} examples, {problem.nnz} nnz, {problem.epochs} epochs, sequential "
                  f"Algorithm-1 SGD in plain C, {dt:.1f} s")
    else:
        rows = int(min(n, max(rows, rows * target_s / max(dt, 1e-6))))
        t0 = time.perf_counter()
        oracle.sgd(problem, epochs=1, rows=rows)
        dt = time.perf_counter() - t0
        nnz = int(problem.row_ptr[rows])
        sample = (f"first {rows} of {n} examples ({nnz} nnz, k~{k_mean:.0f}), 1 epoch, sequential Algorithm-1 SGD "
                  f"in plain C, {dt:.1f} s")
    return {"value": nnz / dt, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample}


def recorded_traffic(kernel: str, workload: str, nnz: int):
    """DRAM bytes per launch from the committed ncu summary of this kernel and
    workload, if the kernel sources still hash as they did when it was taken;
    the record is for a launch over `traffic_nnz` nonzeros and scales to this
    run's nonzeros in proportion (the summary shows the bytes per nonzero
    holding across sizes)."""
    import hashlib
    import re
    path = os.path.join(ROOT, "profiles", f"{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m_b = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    m_n = re.search(r"traffic_nnz:\s*([0-9]+)", text)
    m_h = re.search(r"source_sha256:\s*([0-9a-f]{64})", text)
    if not (m_b and m_n and m_h):
        return None
    h = hashlib.sha256()
    sources = {"k_sgd_window": "window.cu", "k_sgd_chain": "chain.cu"}.get(kernel, "sgd.cu")
    for f in (sources, "common.cuh"):
        with open(os.path.join(ROOT, "paper_1508_00703_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest() != m_h.group(1):
        return None
    return float(m_b.group(1)) * nnz / int(m_n.group(1))


def training_loss(p, X, y, w, torch):
    """Mean loss of the workload over its examples at weights w (a measurement
    with library sparse ops, outside every timed region)."""
    vals = X.val if X.val is not None else torch.ones(p.nnz, dtype=torch.float32, device="cuda")
    A = torch.sparse_csr_tensor(X.row_ptr, X.col.to(torch.int64), vals, size=(p.n_rows, p.n_cols))
    m = torch.mv(A.to(torch.float64), w.to(torch.float64))
    yy = y.to(torch.float64)
    if p.loss == 0:
        return float(torch.nn.functional.softplus(-yy * m).mean())
    if p.loss == 1:
        return float((0.5 * (m - yy) ** 2).mean())
    return float(torch.clamp(1.0 - yy * m, min=0.0).mean())


def workload_config(name, problem, mode):
    import synthdata
    spec = synthdata.WORKLOADS[name]
    desc = (f"{name}: {problem.n_rows} examples x {problem.n_cols} features, {spec['k']} nnz/row "
            f"{spec['ids']}{' s=' + str(spec['zipf_s']) if spec['ids'] == 'zipf' else ''} ids, "
            f"{spec['vals']} values, {spec['loss']} loss, eta={spec['eta']}, {spec['epochs']} epochs")
    in_bytes = problem.nnz * (4 + (0 if problem.val is None else 4)) + 8 * (problem.n_rows + 1)
    return {"workload": desc, "schedule": mode, "epochs": problem.epochs,
            "nnz": problem.nnz, "n_rows": problem.n_rows, "n_cols": problem.n_cols,
            "l2": ("inputs larger than L2: CSR %.2f GB and w %.2f GB vs %d MB L2" %
                   (in_bytes / 1e9, 4 * problem.n_cols / 1e9, L2_BYTES // 2 ** 20)
                   if in_bytes > L2_BYTES else "inputs fit in L2")}


# ---------------------------------------------------------------- our implementation
def run_ours(args, rank, world, local_rank):
    import numpy as np
    import torch

    import synthdata
    import paper_1508_00703_gb300 as pdb

    torch.cuda.set_device(local_rank)
    overrides = {} if args.rows is None else {"n_rows": args.rows}
    p = synthdata.generate(args.workload, seed=synthdata.DATA_SEED + rank, **overrides)
    E = p.epochs
    mode = {"auto": pdb.PDB_SCHED_AUTO, "ready": pdb.PDB_SCHED_READY, "levels": pdb.PDB_SCHED_LEVELS,
            "chain": pdb.PDB_SCHED_CHAIN, "window": pdb.PDB_SCHED_WINDOW}[args.mode]
    X = pdb.Csr.from_problem(p)
    y = torch.from_numpy(p.y).cuda()
    w = torch.zeros(p.n_cols, dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()
    opts = dict(ticket_chunk=args.ticket_chunk, blocks_per_sm=args.blocks_per_sm)

    batch = (p.bsp_batch or 4096) if args.bsp < 0 else args.bsp

    def step():
        w.zero_()
        c = pdb.pdb_build_conflicts(X, stream)
        if batch:
            pdb.pdb_bsp_epoch(X, y, c, w, p.loss, p.eta, batch, E, opts=opts, stream=stream)
            return c, None
        if args.delay is not None:
            s = pdb.pdb_schedule_build(c, pdb.PDB_SCHED_READY, stream)
            gates = pdb.PDB_SSP_PREFIX if args.ssp_gates == "prefix" else pdb.PDB_SSP_COUNT
            pdb.pdb_ssp_epoch(X, y, c, s, w, p.loss, p.eta, E, args.delay, opts=dict(opts, ssp_gates=gates),
                              stream=stream)
            return c, s
        s = pdb.pdb_schedule_build(c, mode, stream)
        pdb.pdb_sgd_epoch(X, y, c, s, w, p.loss, p.eta, E, opts=opts, stream=stream)
        return c, s

    for _ in range(args.warmup):
        c, s = step()
        pdb.check_status(c, stream)
        del c, s

    phases = []
    barrier(world)
    torch.cuda.synchronize()
    launches0 = pdb.pdb_launch_count()
    with ClockSampler(local_rank) as clk:
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        marks = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        ev0.record(stream)
        marks[0].record(stream)
        for i in range(args.steps):
            c, s = step()
            marks[i + 1].record(stream)
            phases.append(pdb.pdb_get_stats(c, s))   # synchronizes; frees the step's handles below
            del c, s
        ev1.record(stream)
        torch.cuda.synchronize()
    per_step = sorted(marks[i].elapsed_time(marks[i + 1]) for i in range(args.steps))
    barrier(world)
    launches = pdb.pdb_launch_count() - launches0
    ms_step = ev0.elapsed_time(ev1) / args.steps
    ms_step = reduce_max(ms_step, world)
    units = E * p.nnz
    total_units = reduce_sum(units, world)
    value = total_units / (ms_step / 1e3)

    # the step's result is checked after timing: parity with the oracle is the tests' job
    c, s = step()
    pdb.check_status(c, stream)
    del c, s

    ms_sgd = statistics.median(ph["ms_bsp" if batch else "ms_sgd"] for ph in phases)
    ms_kern = statistics.median(ph["ms_bsp" if batch else "ms_sgd_kernels"] for ph in phases)
    ms_build = statistics.median(ph["ms_build"] for ph in phases)
    ms_sched = statistics.median(ph["ms_schedule"] for ph in phases)
    peak, peak_kind = measured_peak_hbm()
    sgd_bytes_per_launch = ALG_BYTES_PER_NNZ * p.nnz + ALG_BYTES_PER_ROW * p.n_rows
    sgd_launch_ms = ms_kern / E
    sgd_gbs = sgd_bytes_per_launch / (sgd_launch_ms / 1e3) / 1e9
    resolved = int(phases[0]["sched_mode"])
    if args.delay is not None:
        resolved = -2
    kname = {pdb.PDB_SCHED_READY: "k_sgd_ready", pdb.PDB_SCHED_LEVELS: "k_sgd_levels", -1: "k_bsp", -2: "k_sgd_ssp",
             pdb.PDB_SCHED_CHAIN: "k_sgd_chain", pdb.PDB_SCHED_WINDOW: "k_sgd_window"}[resolved]
    roofline = {"kernel": kname,
                "bound": "hbm", "achieved": round(sgd_gbs, 1), "peak": peak, "unit": "GB/s",
                "frac": round(sgd_gbs / peak, 4), "traffic": recorded_traffic(kname, args.workload, p.nnz),
                "peak_source": peak_kind,
                "algorithmic_bytes_per_launch": sgd_bytes_per_launch, "launch_ms": round(sgd_launch_ms, 4),
                "frac_of_8TBs": round(sgd_gbs / 8000.0, 4)}
    if roofline["traffic"]:
        # the DRAM bytes ncu counted per launch over this run's launch time: how busy
        # HBM is, against the algorithmic fraction above (random 4-byte accesses move
        # whole sectors)
        dram_gbs = roofline["traffic"] / (sgd_launch_ms / 1e3) / 1e9
        roofline["dram_gbs"] = round(dram_gbs, 1)
        roofline["dram_frac"] = round(dram_gbs / peak, 4)
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded generator, no dataset)",
        "config": dict(workload_config(args.workload, p,
                                       f"bsp, mini-batch {batch}" if batch else
                                       f"admissible delay {args.delay} (READY records)" if args.delay is not None else
                                       {0: "levels", 1: "ready", 2: "chain", 4: "window"}[resolved]
                                       + (" (auto)" if args.mode == "auto" else "")),
                       parallelism=f"replicas{world}" if world > 1 else "single GPU",
                       ticket_chunk=args.ticket_chunk or 2),
        "roofline": roofline,
        "phases_ms": ({"build_conflicts": ms_build, "bsp_all_epochs": ms_sgd} if batch else
                      {"build_conflicts": ms_build, "schedule": ms_sched, "sgd_all_epochs": ms_sgd,
                       "sgd_update_kernels": ms_kern}),
        "sgd_only": {"value": units / (ms_sgd / 1e3), "unit": UNIT},
        # per-step device times (the paper's protocol: trimmed mean without the 2 fastest and 2 slowest)
        "step_ms": {"trimmed_mean": statistics.mean(per_step[2:-2] if len(per_step) > 4 else per_step),
                    "median": statistics.median(per_step), "min": per_step[0], "max": per_step[-1]},
        "gpu_launches": int(launches),
        "clocks": clk.summary(),
    }

    if args.delay is not None:
        result["metric"] = METRIC.replace("serially-equivalent sparse SGD",
                                          f"admissible-delay ({args.delay}) sparse SGD")
        result["config"]["ssp_gates"] = args.ssp_gates
        if args.delay > 0:
            result["config"]["note"] = "delay > 0: not serially equivalent, result depends on timing"
        # what the staleness costs: the training loss after the delayed run beside
        # the exact (serially equivalent) run's, both from w = 0 over the same epochs
        c, s = step()
        pdb.check_status(c, stream)
        delayed = training_loss(p, X, y, w, torch)
        w.zero_()
        c2 = pdb.pdb_build_conflicts(X, stream)
        s2 = pdb.pdb_schedule_build(c2, pdb.PDB_SCHED_AUTO, stream)
        pdb.pdb_sgd_epoch(X, y, c2, s2, w, p.loss, p.eta, E, stream=stream)
        pdb.check_status(c2, stream)
        result["training_loss"] = {"delayed": delayed, "exact": training_loss(p, X, y, w, torch),
                                   "loss": {0: "logistic", 1: "squared", 2: "hinge"}[p.loss]}
        del c, s, c2, s2
    if batch:
        roofline["kernel"] = "k_bsp (whole pdb_bsp_epoch call per epoch: batch sort, gather, cooperative kernel)"
        result["metric"] = METRIC.replace("serially-equivalent sparse SGD", f"BSP mini-batch ({batch}) SGD")
        del result["sgd_only"]
        result["bsp_only"] = {"value": units / (ms_sgd / 1e3), "unit": UNIT}
    if not args.no_e2e and not batch and args.delay is None:
        result["e2e"] = run_e2e(args, p, mode, pdb, torch, world)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(p, args.cpu_seconds)
    del np
    return result


def run_e2e(args, p, mode, pdb, torch, world):
    """Same metric through the public API from pinned host buffers: every
    step copies its inputs host-to-device and reads the trained weights back,
    inside the timed region.  The inputs of steps i+1 and i+2 copy on a copy
    stream into two more sets of device buffers while step i computes, and
    step i's weights go back to the host on a third stream while step i+1
    computes (an input pipeline two steps deep, as a training loop that
    streams its data would run it: one copy slowed by the host link then
    delays no step by itself)."""
    # a stream of its own for the compute: the legacy default stream would order
    # itself against the copy streams
    main = torch.cuda.Stream()
    h_row = torch.from_numpy(p.row_ptr).pin_memory()
    h_col = torch.from_numpy(p.col).pin_memory()
    h_val = None if p.val is None else torch.from_numpy(p.val).pin_memory()
    h_y = torch.from_numpy(p.y).pin_memory()
    h_w0 = torch.zeros(p.n_cols, dtype=torch.float32).pin_memory()
    DEPTH = 3                                   # sets of device buffers: step i and the inputs of i+1, i+2
    h_w = [torch.empty(p.n_cols, dtype=torch.float32).pin_memory() for _ in range(DEPTH)]
    h2d = sum(t.numel() * t.element_size() for t in (h_row, h_col, h_val, h_y, h_w0) if t is not None)
    d2h = h_w[0].numel() * h_w[0].element_size()

    class Buffers:
        def __init__(self):
            self.row = torch.empty_like(h_row, device="cuda")
            self.col = torch.empty_like(h_col, device="cuda")
            self.val = None if h_val is None else torch.empty_like(h_val, device="cuda")
            self.y = torch.empty_like(h_y, device="cuda")
            self.w = torch.empty_like(h_w0, device="cuda")
            self.X = pdb.Csr(self.row, self.col, self.val, p.n_cols)
            self.copied = torch.cuda.Event()
            self.done = torch.cuda.Event()       # compute on these buffers finished
            self.read = torch.cuda.Event()       # their weights are back on the host
            self.done.record(main)
            self.read.record(main)

    bufs = [Buffers() for _ in range(DEPTH)]
    copy_in, copy_out = torch.cuda.Stream(), torch.cuda.Stream()

    def stage(i):
        b = bufs[i % DEPTH]
        copy_in.wait_event(b.done)            # step i-DEPTH no longer reads these inputs
        copy_in.wait_event(b.read)            # and its weights have left the device
        with torch.cuda.stream(copy_in):
            for d, h in ((b.row, h_row), (b.col, h_col), (b.val, h_val), (b.y, h_y), (b.w, h_w0)):
                if d is not None:
                    d.copy_(h, non_blocking=True)
            b.copied.record(copy_in)

    def compute(i):
        b = bufs[i % DEPTH]
        main.wait_event(b.copied)
        c = pdb.pdb_build_conflicts(b.X, main)
        s = pdb.pdb_schedule_build(c, mode, main)
        pdb.pdb_sgd_epoch(b.X, b.y, c, s, b.w, p.loss, p.eta, p.epochs,
                          opts=dict(ticket_chunk=args.ticket_chunk, blocks_per_sm=args.blocks_per_sm), stream=main)
        b.done.record(main)
        copy_out.wait_event(b.done)
        with torch.cuda.stream(copy_out):
            h_w[i % DEPTH].copy_(b.w, non_blocking=True)
            b.read.record(copy_out)
        return c, s

    phases = []

    def run(steps):
        for i in range(min(DEPTH - 1, steps)):
            stage(i)
        for i in range(steps):
            if i + DEPTH - 1 < steps:
                stage(i + DEPTH - 1)
            c, s = compute(i)
            rc = pdb.pdb_status(c, main)        # synchronizes main: step i's kernels are done
            if rc != 0:
                raise pdb.PdbError(rc, "e2e step")
            phases.append(pdb.pdb_get_stats(c, s))   # the step's device phases (CUDA events)
            del c, s
        copy_out.synchronize()                  # the last step's weights are on the host

    steps = max(2, min(args.steps, 10))
    run(2)
    phases.clear()
    # the host link's bandwidth on this machine, for reading the number (after the
    # warm-up steps; best of two copies each way)
    link = {}
    for name, dst, src in (("h2d_gbs", bufs[0].col, h_col), ("d2h_gbs", h_w[0], bufs[0].w)):
        best = 0.0
        for _ in range(2):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(copy_in)
            with torch.cuda.stream(copy_in):
                dst.copy_(src, non_blocking=True)
            e1.record(copy_in)
            e1.synchronize()
            best = max(best, src.numel() * src.element_size() / (e0.elapsed_time(e1) / 1e3) / 1e9)
        link[name] = round(best, 1)
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    run(steps)
    torch.cuda.synchronize()
    dt = (time.perf_counter() - t0) / steps
    dt = reduce_max(dt, world)
    units = reduce_sum(p.epochs * p.nnz, world)
    return {"value": units / dt, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": dt * 1e3, "steps": steps, "host_link": link,
            "device_phases_ms": {"build_conflicts": statistics.median(ph["ms_build"] for ph in phases),
                                 "sgd_all_epochs": statistics.median(ph["ms_sgd"] for ph in phases)},
            "pipeline": "steps i+1 and i+2's H2D on a copy stream and step i's D2H on another, overlapping the next step"}


# ---------------------------------------------------------------- reference arm: the CPU oracle
def run_reference(args, rank, world):
    import synthdata
    import oracle

    overrides = {} if args.rows is None else {"n_rows": args.rows}
    p = synthdata.generate(args.workload, **overrides)
    n = p.n_rows
    per_step_s = max(1.0, min(10.0, 150.0 / max(1, args.steps + args.warmup)))
    rows = min(n, 20000)
    t0 = time.perf_counter()
    oracle.sgd(p, epochs=1, rows=rows)
    dt = time.perf_counter() - t0
    rows = int(min(n, max(rows, rows * per_step_s / max(dt, 1e-6))))
    for _ in range(args.warmup):
        oracle.sgd(p, epochs=1, rows=rows)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.sgd(p, epochs=1, rows=rows)
        times.append(time.perf_counter() - t0)
    nnz = int(p.row_ptr[rows])
    ms = 1e3 * sum(times) / len(times)
    value = nnz / (ms / 1e3)
    sample = (f"first {rows} of {n} examples ({nnz} nnz), 1 epoch per step, sequential Algorithm-1 SGD "
              f"in plain C on 1 host core")
    cfg = workload_config(args.workload, p, "sequential")
    return {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded generator, no dataset)",
            "config": cfg,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main(argv=None):
    args = parse_args(argv)
    rank, world, local_rank = dist_env()
    if args.impl == "reference":
        if rank != 0:
            return 0
        print(json.dumps(run_reference(args, rank, world)), flush=True)
        return 0
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local_rank)
        dist.init_process_group(backend=backend)
    result = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
