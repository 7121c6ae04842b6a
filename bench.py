#!/usr/bin/env python
"""Benchmark of the MeqMuon optimizer step (all 2D hidden weights of a model).

Metric: milliseconds per optimizer step for the whole model (lower is
better), with NS TFLOP/s and the bandwidth kernels' GB/s as fractions of the
measured GB300 peaks.

Default workload: the Llama-7B-class hidden weights (32 layers, d 4096, ffn
11008: 224 matrices, 6.48G elements; params + grads + momentum 77.7 GB on
one GPU), the largest single-GPU configuration; seeded synthetic gradients
(see paper_2609_35701_gb300/workloads.py). Every workload's state is larger
than L2, so no flush is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--layers L]
  python bench.py --impl reference ...   # the fp64 CPU oracle on host cores

With N > 1 (torchrun), the matrices are split across ranks (flop-balanced,
no data-path collective); the time is the max over ranks.
"""
from __future__ import annotations

import argparse
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

LR, MU, WD, EPS = 0.02, 0.95, 0.1, 1e-7
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
BW_BYTES_PER_ELEM = 24  # read G, B; write B; write X_0 (2 B); read U (2 B); read + write W
REFERENCE_BUDGET_S = 150.0   # wall-clock budget of all oracle samples of --impl reference
CPU_BASELINE_BUDGET_S = 20.0 # wall-clock budget of the oracle sample beside the GPU line
SUSTAINED_NS_MS = 20.0       # an NS phase this long per step runs under the power cap: sustained peak
DEFAULT_STEPS = {"llama7b": 20, "llama1b": 50}
METRIC = "MeqMuon step ms per model; NS TFLOP/s & equilibration GB/s as % of GB300 peak"
COPY_CHUNK = 8 << 20          # smallest piece (elements, 32 MB) of a host <-> device copy in the end-to-end loop
COPY_PIECES = 64              # at most this many pieces per direction per step


def source_fingerprint(path):
    """sha256 prefix of a C++/CUDA source with comments and whitespace removed
    (so that an edit to a comment does not detach a recorded measurement)."""
    import hashlib
    import re

    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    text = re.sub(r"\s+", "", text)
    return hashlib.sha256(text.encode()).hexdigest()[:16]


def recorded_traffic(workload):
    """dram read + write bytes per ns_gemm launch from the committed ncu
    summary, if the kernel source is unchanged since that capture."""
    import hashlib
    import re

    path = os.path.join(ROOT, "profiles", f"ns_gemm_{workload}.md")
    src = os.path.join(ROOT, "paper_2609_35701_gb300", "csrc", "ns_gemm.cu")
    try:
        text = open(path).read()
        sha = source_fingerprint(src)
        m = re.search(r"code fingerprint `([0-9a-f]+)`", text)
        t = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+-]+)", text)
        if m and t and m.group(1) == sha:
            return float(t.group(1))
    except Exception:
        pass
    return None


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


def ns_flops(s, l, K):
    """Algorithmic NS flops of one matrix (Eq. (5), K iterations), counting
    the symmetric halves of A = X X^T and A^2 once, and the dense count."""
    sym = K * (s * (s + 1) * l + s * s * (s + 1) + 2 * s * s * l)
    dense = K * (4 * s * s * l + 2 * s * s * s)
    return sym, dense


def partition(shapes, world, K=5, kinds=None):
    """Greedy flop-balanced split of matrix indices over ranks (entries that
    are not hidden weights carry no NS work and are weighted by size)."""
    kinds = kinds or [0] * len(shapes)
    w = [(ns_flops(min(r, c), max(r, c), K)[0] if k == 0 else 24 * r * c, i)
         for i, ((r, c), k) in enumerate(zip(shapes, kinds))]
    w.sort(reverse=True)
    load = [0] * world
    parts = [[] for _ in range(world)]
    for f, i in w:
        k = min(range(world), key=lambda j: load[j])
        parts[k].append(i)
        load[k] += f
    return [sorted(p) for p in parts]


class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons."""

    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits", "-lms", "50",
                 "-i", str(self.gpu_id)], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.12)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[5 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def oracle_flops(r, c, kind, K=5):
    """fp64 flops of the oracle's step for one (rows, cols) matrix: Eq. (5)
    as written (A = X X^T on the row side, A A, then (b A + c A^2) X), or a
    few dozen per element for the branches without Newton-Schulz."""
    if kind != 0:
        return 30 * r * c
    return K * (4 * r * r * c + 2 * r ** 3)


def oracle_sample(wl, seed_step=0, rule="meqmuon", budget_s=None):
    """Times the fp64 oracle on one matrix of each (rows, cols, kind) class of
    the workload, cheapest first, and extrapolates to the whole model step
    (ms). With a budget, a class whose predicted time (the flop rate of the
    classes timed so far) would overrun it is not run: its time is that rate
    times its flop count. Returns (ms, timed classes, estimated classes)."""
    import numpy as np

    from oracle import meqmuon as O
    from paper_2609_35701_gb300 import workloads as W

    classes = {}
    kinds = wl.kind_list()
    for i, (_, r, c) in enumerate(wl.shapes):
        classes.setdefault((r, c, kinds[i]), []).append(i)
    order = sorted(classes, key=lambda k: oracle_flops(*k))
    total_ms, spent, flops_done = 0.0, 0.0, 0.0
    timed, estimated = [], []

    def label(r, c, k):
        return f"{r}x{c}" + ("" if k == 0 else ("/2-sided" if k == 1 else "/vector"))

    for (r, c, k) in order:
        idx = classes[(r, c, k)]
        f = oracle_flops(r, c, k)
        if timed and budget_s is not None and spent > 0 and spent + f / (flops_done / spent) > budget_s:
            total_ms += f / (flops_done / spent) * 1e3 * len(idx)
            estimated.append(label(r, c, k))
            continue
        G = W.gradient(wl, idx[0], seed_step).double().numpy()
        W0 = np.zeros((r, c))
        Bp = np.zeros((r, c))
        t0 = time.perf_counter()
        if rule == "muon":
            O.moonlight_step(W0, G, Bp, LR, MU, WD)
        else:
            O.param_step(k, W0, G, Bp, LR, MU, WD, eps=EPS)
        dt = time.perf_counter() - t0
        spent += dt
        flops_done += f
        total_ms += dt * 1e3 * len(idx)
        timed.append(label(r, c, k))
    return total_ms, timed, estimated


def sample_text(wl, timed, estimated, repeats):
    t = (f"fp64 oracle on one matrix per shape class, timed: {', '.join(timed)}"
         + (f"; estimated from the timed classes' flop rate x the oracle's own flop count: {', '.join(estimated)}"
            if estimated else "")
         + f"; {repeats} sample(s); extrapolated by class counts to all {len(wl.shapes)} matrices")
    return t


def workload_for(args):
    from paper_2609_35701_gb300 import workloads as W

    wl = W.get_workload(args.workload)
    return W.first_layers(wl, args.layers) if args.layers else wl


def cpu_cores():
    try:
        n = len(os.sched_getaffinity(0))
    except Exception:
        n = os.cpu_count() or 1
    for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(v, "").isdigit():
            n = min(n, int(os.environ[v]))
    return n


def run_reference(args):
    """--impl reference: the fp64 CPU oracle, as it stands, on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    wl = workload_for(args)
    # each sample gets an equal share of the budget (the warm-up sample too),
    # so the whole --steps K --warmup W run stays within a few minutes
    per = max(REFERENCE_BUDGET_S / (args.steps + 1), 2.0)
    oracle_sample(wl, 0, rule=args.update_rule, budget_s=per)  # warm-up (BLAS threads)
    vals = []
    timed = estimated = None
    t0 = time.perf_counter()
    for k in range(args.steps):
        ms, timed, estimated = oracle_sample(wl, k, rule=args.update_rule, budget_s=per)
        vals.append(ms)
        if time.perf_counter() - t0 > REFERENCE_BUDGET_S:
            break  # the samples are timed on the host cores: keep the whole run to a few minutes
    v = statistics.median(vals)
    cores = cpu_cores()
    sample = sample_text(wl, timed, estimated, len(vals)) + " (one sample per step)"
    line = {
        "impl": "reference", "metric": METRIC, "value": v,
        "unit": "ms/step", "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": v, "higher_is_better": False, "scaling": "strong", "vs_baseline": None, "dtype": "f64",
        "timed_steps": len(vals), "data": "synthetic", "config": {"workload": wl.name, "matrices": len(wl.shapes), "elements": wl.numel,
                                        "update_rule": "Eq. (11) + Eq. (14)" if args.update_rule == "meqmuon" else "Eq. (6)"},
        "cpu_baseline": {"value": v, "unit": "ms/step", "cores": cores, "kind": "oracle", "sample": sample},
        "e2e": {"value": v, "unit": "ms/step", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_trajectory(args):
    """Times meq_ns_cv_trajectory (one matrix of every hidden shape of the
    workload, gradients of step 0) and the fp64 oracle's replay of the same
    matrices on the host cores. One JSON line."""
    import numpy as np
    import torch

    import __graft_entry__

    __graft_entry__.build()
    from oracle import meqmuon as O
    from paper_2609_35701_gb300 import meq
    from paper_2609_35701_gb300 import workloads as W

    wl = workload_for(args)
    kinds = wl.kind_list()
    firsts = {}
    for i, (_, r, c) in enumerate(wl.shapes):
        if kinds[i] == W.HIDDEN:
            firsts.setdefault((r, c), i)
    Hs = {rc: W.gradient(wl, i, 0) for rc, i in firsts.items()}
    dev = {rc: h.cuda().contiguous() for rc, h in Hs.items()}
    K = args.ns_trajectory
    for _ in range(2):
        for h in dev.values():
            meq.ns_cv_trajectory(h, steps=K)
    torch.cuda.synchronize()
    reps = max(1, min(args.steps, 5))
    t0 = time.perf_counter()
    for _ in range(reps):
        for h in dev.values():
            meq.ns_cv_trajectory(h, steps=K)
    gpu_ms = (time.perf_counter() - t0) * 1e3 / reps
    t0 = time.perf_counter()
    for h in Hs.values():
        O.ns_cv_trajectory(h.double().numpy(), steps=K)
    cpu_ms = (time.perf_counter() - t0) * 1e3
    shapes = ", ".join(f"{r}x{c}" for r, c in Hs)
    line = {
        "metric": f"NS CV trajectory replay, k = 0..{K} (Section 3.1)", "value": gpu_ms, "unit": "ms (all shapes)",
        "n_gpus": 1, "steps": reps, "warmup": 2, "higher_is_better": False, "dtype": "fp16", "data": "synthetic",
        "config": {"workload": wl.name, "shapes": shapes,
                   "method": "one state per k (ns_steps = k) through the CUDA step, k = 0 by the statistics kernel"},
        "cpu_baseline": {"value": cpu_ms, "unit": "ms (all shapes)", "cores": cpu_cores(), "kind": "oracle",
                         "sample": f"fp64 oracle replay of the same {len(Hs)} matrices"},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None, help="timed steps (default: 20 for llama7b, 50 for llama1b, "
                    "200 otherwise)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama7b")
    ap.add_argument("--layers", type=int, default=0,
                    help="use only the first L layers of the workload (a smaller case of the same kernels)")
    ap.add_argument("--ns-fp16-mask", type=lambda x: int(x, 0), default=0xFFFFFFFF)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--update-rule", default="meqmuon", choices=["meqmuon", "muon"],
                    help="meqmuon: Eq. (11) + Eq. (14); muon: the Eq. (6) comparison baseline (hidden weights only)")
    ap.add_argument("--ns-trajectory", type=int, default=0, metavar="K",
                    help="instead of the step, time the Section 3.1 CV replay of X_0..X_K (one matrix per shape)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    if args.steps is None:
        args.steps = DEFAULT_STEPS.get(args.workload, 200)
    if args.impl == "reference":
        run_reference(args)
        return
    if args.ns_trajectory:
        run_trajectory(args)
        return

    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    import __graft_entry__

    __graft_entry__.build()
    from paper_2609_35701_gb300 import meq
    from paper_2609_35701_gb300 import workloads as W

    wl = workload_for(args)
    mine = partition([(r, c) for _, r, c in wl.shapes], world, kinds=wl.kind_list())[rank]
    shapes = [(wl.shapes[i][1], wl.shapes[i][2]) for i in mine]
    all_kinds = wl.kind_list()
    kinds = [all_kinds[i] for i in mine]
    dev = torch.device("cuda", local)

    # Flat, 256-byte aligned device buffers with one view per matrix.
    def flat_views(nums, device, pin=False):
        offs, tot = [], 0
        for n in nums:
            offs.append(tot)
            tot += (n + 63) // 64 * 64
        if device == "cpu":
            buf = torch.empty(tot, dtype=torch.float32, pin_memory=pin)
        else:
            buf = torch.empty(tot, dtype=torch.float32, device=device)
        return buf, [buf[o:o + n] for o, n in zip(offs, nums)]

    nums = [r * c for r, c in shapes]
    pbuf, pviews = flat_views(nums, dev)
    gbufs = []
    for t in range(2):
        gb, gv = flat_views(nums, dev)
        for j, i in enumerate(mine):
            gv[j].copy_(W.gradient(wl, i, t, device=dev).reshape(-1))
        gbufs.append((gb, gv))
    w0 = W.initial_weights(wl, device=dev)
    for j, i in enumerate(mine):
        pviews[j].copy_(w0[i].reshape(-1))
    del w0
    params = [v.view(r, c) for v, (r, c) in zip(pviews, shapes)]
    grads = [[v.view(r, c) for v, (r, c) in zip(gv, shapes)] for _, gv in gbufs]

    rule = meq.RULE_MUON if args.update_rule == "muon" else meq.RULE_MEQMUON
    opt = meq.MeqMuon(shapes, kinds=kinds, ns_fp16_mask=args.ns_fp16_mask, update_rule=rule)
    stream = torch.cuda.current_stream()
    for k in range(args.warmup):
        opt.step(params, grads[k % 2], LR, MU, WD, EPS)
    opt.sync()

    props = torch.cuda.get_device_properties(local)
    gpu_id = getattr(props, "uuid", None)
    gpu_id = f"GPU-{gpu_id}" if gpu_id is not None and not str(gpu_id).startswith("GPU-") else (gpu_id or local)
    clocks = ClockSampler(gpu_id)
    clocks.start()
    time.sleep(0.15)
    # ---------------- timed region: K steps, CUDA events on the launch stream
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for k in range(args.steps):
        opt.step(params, grads[k % 2], LR, MU, WD, EPS)
    e1.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clk = clocks.stop()
    opt.sync()
    ms = e0.elapsed_time(e1) / args.steps
    if world > 1:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())

    # ---------------- per-phase timing (events between phases, eager launches)
    opt.set_profiling(True)
    for k in range(args.steps):
        opt.step(params, grads[k % 2], LR, MU, WD, EPS)
    phases, nprof = opt.read_profile()
    opt.set_profiling(False)
    ph = {k: v / max(nprof, 1) for k, v in phases.items()}

    K = 5
    hid = [sh for sh, k in zip(shapes, kinds) if k == W.HIDDEN]   # Newton-Schulz runs on hidden weights only
    sym = sum(ns_flops(min(r, c), max(r, c), K)[0] for r, c in hid)
    dense = sum(ns_flops(min(r, c), max(r, c), K)[1] for r, c in hid)
    n_gemm_launches = opt.ns_gemm_launches_per_step
    peaks, peak_src = load_peaks()
    # an NS phase that runs tens of milliseconds at a time draws the power
    # cap: its denominator is the sustained bf16 figure, else the burst one
    sustained = ph["ns_gemm"] >= SUSTAINED_NS_MS
    ns_peak = peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"]
    ns_tflops = sym / (ph["ns_gemm"] * 1e-3) / 1e12
    ns_dense_tflops = dense / (ph["ns_gemm"] * 1e-3) / 1e12
    numel = sum(nums)
    # algorithmic bytes of the bandwidth phases: 24 B / element, plus the
    # column pass over the momentum (4 B) for the remaining 2D parameters
    bw_bytes = sum((BW_BYTES_PER_ELEM + (4 if k == W.REMAINING_2D else 0)) * r * c for (r, c), k in zip(shapes, kinds))
    bw_ms = ph["momentum"] + ph["cast_x0"] + ph["stats"] + ph["apply"]
    bw_gbs = bw_bytes / (bw_ms * 1e-3) / 1e9

    # ---------------- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        # one pinned host copy of the gradients serves both device buffers
        # (every step uploads a whole gradient set; at Llama-7B one set is
        # 25.9 GB, so two would pin another 26 GB of host memory)
        h = torch.empty(gbufs[0][0].numel(), dtype=torch.float32, pin_memory=True)
        h.copy_(gbufs[0][0])
        hg = [h, h]
        hp = torch.empty(pbuf.numel(), dtype=torch.float32, pin_memory=True)
        n_e2e = max(3, min(args.steps, 50))
        # Copies move in pieces on two copy streams, so that the two
        # directions share the host link: the gradients of step k + 1 go up
        # while step k runs (enqueued right after step k's prepare); the
        # parameters of step k - 1 come back while step k's momentum,
        # Newton-Schulz and statistics run (meq_step_prepare), and step k's
        # update (meq_step_apply) waits for that copy before it writes the
        # parameters in place. At most COPY_PIECES pieces per direction keep
        # the host from blocking on a full queue of pending copies.
        chunk = max(COPY_CHUNK, -(-pbuf.numel() // COPY_PIECES))
        pieces = [(lo, min(lo + chunk, pbuf.numel())) for lo in range(0, pbuf.numel(), chunk)]
        up, down = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
        ev_in = [torch.cuda.Event() for _ in range(2)]
        ev_prep = [torch.cuda.Event() for _ in range(2)]
        ev_step = torch.cuda.Event()
        ev_out = torch.cuda.Event()

        def upload(k):
            b = k % 2
            with torch.cuda.stream(up):
                if k >= 2:
                    up.wait_event(ev_prep[b])   # step k - 2 has read this gradient buffer
                for lo, hi in pieces:
                    gbufs[b][0][lo:hi].copy_(hg[b][lo:hi], non_blocking=True)
                ev_in[b].record(up)

        torch.cuda.synchronize()
        a0 = torch.cuda.Event(enable_timing=True)
        a1 = torch.cuda.Event(enable_timing=True)
        a0.record(stream)
        up.wait_event(a0)
        upload(0)
        for k in range(n_e2e):
            b = k % 2
            stream.wait_event(ev_in[b])
            opt.step_prepare(grads[b], LR, MU, WD, EPS)
            ev_prep[b].record(stream)
            if k + 1 < n_e2e:
                upload(k + 1)
            if k >= 1:
                stream.wait_event(ev_out)        # parameters of step k - 1 are back on the host
            opt.step_apply(params)
            ev_step.record(stream)
            with torch.cuda.stream(down):
                down.wait_event(ev_step)
                for lo, hi in pieces:
                    hp[lo:hi].copy_(pbuf[lo:hi], non_blocking=True)
                ev_out.record(down)
        stream.wait_event(ev_out)
        a1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = a0.elapsed_time(a1) / n_e2e
        if world > 1:
            t = torch.tensor([e2e_ms], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_ms = float(t.item())
        numel_job = numel   # elements of every rank's matrices: the whole job's copies
        if world > 1:
            t = torch.tensor([float(numel)], dtype=torch.float64, device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.SUM)
            numel_job = int(t.item())
        e2e = {"value": e2e_ms, "unit": "ms/step", "h2d_bytes_per_step": 4 * numel_job,
               "d2h_bytes_per_step": 4 * numel_job, "steps": n_e2e,
               "api": "meq_step_prepare + meq_step_apply (parameter read-back of step k - 1 overlaps step k's prepare)"}
    opt.sync()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        vals = []
        t_start = time.perf_counter()
        while True:
            left = CPU_BASELINE_BUDGET_S - (time.perf_counter() - t_start)
            v, timed, estimated = oracle_sample(wl, len(vals), rule=args.update_rule, budget_s=max(left, 1.0))
            vals.append(v)
            if time.perf_counter() - t_start > CPU_BASELINE_BUDGET_S / 2 or len(vals) >= 5:
                break
        cpu = {"value": statistics.median(vals), "unit": "ms/step", "cores": cpu_cores(), "kind": "oracle",
               "sample": sample_text(wl, timed, estimated, len(vals))}

    if rank == 0:
        line = {
            "metric": METRIC,
            "value": ms, "unit": "ms/step", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms, "higher_is_better": False, "scaling": "strong", "vs_baseline": None,
            "dtype": "fp16" if args.ns_fp16_mask == 0xFFFFFFFF else ("bf16" if args.ns_fp16_mask == 0 else "bf16/fp16"),
            "data": "synthetic",
            "config": {"workload": wl.name, "matrices": len(wl.shapes), "elements": wl.numel,
                       "ns_steps": K, "ns_operands": "fp16" if args.ns_fp16_mask == 0xFFFFFFFF else hex(args.ns_fp16_mask),
                       "accumulate": "fp32", "l2": "inputs larger than L2 (params+grads+momentum %.2f GB)" % (12 * wl.numel / 1e9),
                       "parallelism": f"matrices split over {world} GPU(s)" if world > 1 else "single GPU",
                       "update_rule": "Eq. (11) + Eq. (14)" if args.update_rule == "meqmuon" else "Eq. (6)",
                       "ns_launches_per_step": n_gemm_launches},
            "roofline": {
                "bound": "tensor", "kernel": "ns_gemm_kernel",
                "achieved": ns_tflops, "peak": ns_peak, "unit": "TFLOP/s",
                "frac": ns_tflops / ns_peak,
                "peak_source": (f"{peak_src} bf16 dense {'sustained' if sustained else 'burst'} (fp16 rate = bf16 rate;"
                                f" NS phase {ph['ns_gemm']:.2f} ms per step)"),
                "frac_of_burst": ns_tflops / peaks["bf16_tflops"],
                "traffic": recorded_traffic(wl.name),
                "flops_per_launch": sym / max(n_gemm_launches, 1),
                "avg_launch_ms": ph["ns_gemm"] / max(n_gemm_launches, 1),
                "dense_equivalent_tflops": ns_dense_tflops,
            },
            "bandwidth_kernels": {
                "bound": "hbm", "achieved": bw_gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": bw_gbs / peaks["hbm_gbs"], "bytes_per_step": bw_bytes,
                "phase_ms": {k: round(v, 4) for k, v in ph.items()},
            },
            "gpu_launches": opt.kernels_per_step * args.steps,
            "kernels_per_step": opt.kernels_per_step,
            "clocks": clk,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    opt.close()
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
