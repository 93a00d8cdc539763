#!/usr/bin/env python
"""Benchmark of the fused AL8+UF8 AdamW optimizer step on the TinyLlama-1.1B
parameter set (201 tensors, 1,100,048,384 fp32 parameters, blocks of 256).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

One step is one launch of the fused multi-tensor kernel over every tensor.
Inputs are synthetic (seeded device draws: params N(0, 0.02), norm vectors
1.0, grads N(0, 1e-3) with 1% exact zeros; two gradient sets alternate). The
step moves 17.7 GB, far more than L2, so no flush is needed between steps.
Prints one JSON line: params/s (whole job), the roofline of the fused kernel
against the measured HBM copy bandwidth, the CPU oracle on a bounded sample,
an end-to-end figure with host buffers (host<->device copies inside the timed
region), SM clocks sampled during the timed region, and the kernel launch
count. With N > 1 (torchrun) every rank runs an independent replica (the
AdamW step has no cross-rank exchange); value = params of all ranks / max
rank time. --impl reference times the CPU oracle instead (the reference arm).
The same default run then times the other hot-path rows (Adafactor 4096 x
4096, CAME 22 x 2048 x 5632, APOLLO over the 154 TinyLlama matrices, the
AL8/UF8 codec on 2^28 elements) and reports them under "rows", each with its
own clock record, an L2 flush between timed steps and the oracle on a
bounded sample (--no-rows skips them). --workload adafactor|came|apollo|codec
times one of those rows alone, as its own JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = ("optimizer-step params/sec and achieved HBM GB/s (% of GB300 peak), "
          "AL8+UF8 AdamW")
UNIT = "params/s"
KERNEL_SOURCES = ["paper_2608_22322_gb300/csrc/alq_adamw.cu",
                  "paper_2608_22322_gb300/csrc/alq_kernels.cuh",
                  "paper_2608_22322_gb300/csrc/alq_numerics.h"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "adamw_fused_tinyllama.md")
HP = None  # filled in main (needs numpy)
MATS = 0  # --mats: CAME and APOLLO rows on their first K matrices


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--tensors", type=int, default=0,
                    help="use only the first N TinyLlama tensors (profiling runs)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--v-block", type=int, default=256,
                    help="AdamW second-moment block size (256 is the benchmark's "
                         "configuration; 2048 is the paper's core AdamW setting)")
    ap.add_argument("--mats", type=int, default=0,
                    help="CAME and APOLLO rows: only the first K matrices (profiling runs)")
    ap.add_argument("--no-rows", action="store_true",
                    help="skip the other hot-path rows after the headline step")
    ap.add_argument("--workload", default="adamw",
                    choices=["adamw", "adafactor", "came", "apollo", "codec"],
                    help="adamw: the headline TinyLlama AdamW step (default); the others "
                         "time the remaining hot-path rows, one JSON line each")
    return ap.parse_args()


def kernel_sha() -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic():
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources (else None)."""
    try:
        text = open(TRAFFIC_FILE).read()
    except OSError:
        return None
    sha = re.search(r"kernel_sources_sha256:\s*([0-9a-f]+)", text)
    tr = re.search(r"dram_bytes_per_full_launch:\s*([0-9.eE+]+)", text)
    if not sha or not tr or sha.group(1) != kernel_sha():
        return None
    return float(tr.group(1))


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0}, "fallback"


def host_info():
    """The host cores the CPU baselines run on: nproc and the CPU model."""
    model = None
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                model = line.split(":", 1)[1].strip()
                break
    except (OSError, subprocess.SubprocessError):
        pass
    if model is None:
        try:
            for line in open("/proc/cpuinfo"):
                if line.lower().startswith(("model name", "cpu part")):
                    model = line.split(":", 1)[1].strip()
                    break
        except OSError:
            pass
    return {"nproc": os.cpu_count(), "cpu_model": model}


def oracle_threads(ora, want: bool) -> int:
    """Switch the oracle to its OpenMP build (all host cores, the same
    results bit for bit) or back; returns the thread count in use."""
    return ora.use_threads(want)


class ClockSampler:
    """nvidia-smi samples of the GPU's SM clock and throttle reasons."""

    FIELDS = ("uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str):
        self.uuid = uuid
        self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self.file, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.file.flush()
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9 or (self.uuid and self.uuid not in parts[0]):
                    continue
                rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# ------------------------------------------------------- multi-rank -------
def max_over_ranks(ms, device=None):
    """The slowest rank's time: the whole job ends with it. Identity without
    an initialized process group of more than one rank."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return ms
    tt = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def job_value(units_per_rank, world, ms_step):
    """Whole-job throughput: the units every rank processed (each rank runs
    its own replica of the workload: weak scaling) over the slowest rank's
    step time."""
    return units_per_rank * world / (ms_step * 1e-3)


# ------------------------------------------------------------ workload ------
def make_workload(torch, wl, B, n_tensors, dev, v_block=None):
    cfg = wl.CONFIGS["tinyllama_adamw"]
    mb, vb = cfg["m_block"], v_block or cfg["v_block"]
    tens = wl.tinyllama_tensors()
    if n_tensors:
        tens = tens[:n_tensors]
    arrs = []
    for i, (_, shape) in enumerate(tens):
        n = wl.numel(shape)
        p = torch.empty(n, dtype=torch.float32, device=dev)
        if len(shape) == 1:
            p.fill_(1.0)
        else:
            wl.torch_device_normal_(p, 0.02, 1000 + i)
        gs = []
        for k in range(2):
            g = torch.empty(n, dtype=torch.float32, device=dev)
            wl.torch_device_normal_(g, cfg["grad_std"], 50_000 + 7919 * k + i)
            wl.torch_device_zero_(g, cfg["zero_frac"], 90_000 + 7919 * k + i)
            gs.append(g)
        arrs.append(dict(p=p, gs=gs,
                         m_codes=torch.zeros(n, dtype=torch.int8, device=dev),
                         m_absmax=torch.zeros((n + mb - 1) // mb, dtype=torch.float32, device=dev),
                         v_codes=torch.zeros(n, dtype=torch.uint8, device=dev),
                         v_meta=torch.zeros(2 * ((n + vb - 1) // vb), dtype=torch.float32,
                                            device=dev)))
    plans = []
    for k in range(2):
        plans.append(B.AdamWPlan([dict(p=a["p"], g=a["gs"][k], m_codes=a["m_codes"],
                                       m_absmax=a["m_absmax"], v_codes=a["v_codes"],
                                       v_meta=a["v_meta"]) for a in arrs], mb, vb, 8, device=dev))
    n_params = sum(a["p"].numel() for a in arrs)
    return tens, arrs, plans, n_params


def algorithmic_bytes(arrs):
    """p read+write 8, g 4, m and v codes read+write 2, block metadata
    read+write (absmax 4+4 per M block, (l_min, Delta) 8+8 per V block)."""
    tot = 0
    for a in arrs:
        n = a["p"].numel()
        tot += 16 * n + 8 * a["m_absmax"].numel() + 16 * (a["v_meta"].numel() // 2)
    return tot


def cpu_baseline(torch, ora, arrs, hp, t, v_block=256):
    """The oracle on the host cores: its OpenMP build (parallel over blocks
    and elements; the same results as the single-threaded build) over the
    whole parameter set for one step, or, where the compiler has no OpenMP,
    the single-threaded build over the first tensors (up to 180M
    parameters)."""
    threads = oracle_threads(ora, True)
    max_params = None if threads > 1 else 180_000_000
    sample, taken = [], 0
    for a in arrs:
        n = a["p"].numel()
        if max_params is not None and taken + n > max_params and taken > 0:
            break
        sample.append(a)
        taken += n
    host = [dict(p=a["p"].cpu().numpy().copy(), g=a["gs"][0].cpu().numpy(),
                 mc=a["m_codes"].cpu().numpy().copy(), ma=a["m_absmax"].cpu().numpy().copy(),
                 vc=a["v_codes"].cpu().numpy().copy(), vm=a["v_meta"].cpu().numpy().copy())
            for a in sample]
    t0 = time.perf_counter()
    for h in host:
        ora.adamw_step(h["p"], h["g"], h["mc"], h["ma"], h["vc"], h["vm"], 256, v_block, 8, hp, t)
    dt = time.perf_counter() - t0
    oracle_threads(ora, False)
    what = ("all" if len(sample) == len(arrs) else f"the first {len(sample)}")
    return dict({"value": taken / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
                 "sample": f"one step over {what} TinyLlama tensors ({taken} params, {dt:.1f} s "
                           f"on {threads} thread{'s' if threads > 1 else ''})"}, **host_info())


def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    from paper_2608_22322_gb300 import build_lib
    build_lib.build()
    from paper_2608_22322_gb300 import binding as B
    from paper_2608_22322_gb300 import workloads as wl

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local if world > 1 else 0)
    hp = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01,
              log_floor=float(np.float32(np.log2(1e-16))))

    tens, arrs, plans, n_params = make_workload(torch, wl, B, args.tensors, dev, args.v_block)
    nbytes = algorithmic_bytes(arrs)
    stream = torch.cuda.current_stream(dev)
    t = 0
    for _ in range(args.warmup):
        t += 1
        plans[t % 2].step(hp, t)
    torch.cuda.synchronize(dev)

    props = torch.cuda.get_device_properties(dev)
    uuid = str(getattr(props, "uuid", "") or "")
    sampler = ClockSampler(uuid.replace("GPU-", ""))
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        t += 1
        plans[t % 2].step(hp, t)
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    if world > 1:
        dist.barrier()
    ms = ev0.elapsed_time(ev1)
    clocks = sampler.stop()
    ms = max_over_ranks(ms, dev)
    ms_step = ms / args.steps
    launches = args.steps  # one fused kernel launch per step

    peaks, peak_src = measured_peaks()
    achieved = nbytes / (ms_step * 1e-3) / 1e9
    peak = float(peaks.get("hbm_gbs", 6800.0))
    traffic = recorded_traffic() if not args.tensors and args.v_block == 256 else None

    # The other rows next, before the end-to-end and CPU legs (so that no
    # host-side work of those legs is still settling while short steps are
    # timed); single-GPU measurements of their own workloads.
    rows = None
    if rank == 0 and world == 1 and not args.no_rows and not args.tensors:
        import gc
        rows = {}
        for name in ("adafactor", "came", "apollo", "codec"):
            rows[name] = measure_row(name, args, dev, warmup=5, min_steps=20,
                                     with_cpu=not args.no_cpu, summary=True)
            gc.collect()
            torch.cuda.empty_cache()

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(torch, B, arrs, hp, t, args.e2e_steps, n_params, dev)
        t += e2e.pop("_steps_done")
        # whole job: every rank's replica over the slowest rank's time
        e2e["ms_per_step"] = max_over_ranks(e2e["ms_per_step"], dev)
        e2e["value"] = job_value(n_params, world, e2e["ms_per_step"])
        st = e2e["staged"]
        st["ms_per_step"] = max_over_ranks(st["ms_per_step"], dev)
        st["value"] = job_value(n_params, world, st["ms_per_step"])

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        import oracle as ora
        cpu = cpu_baseline(torch, ora, arrs, hp, t + 1, v_block=args.v_block)


    if world > 1:
        dist.destroy_process_group()
    if rank != 0:
        return
    name = "tinyllama-1.1b" if not args.tensors else f"tinyllama-1.1b first {args.tensors} tensors"
    line = {
        "metric": METRIC, "value": job_value(n_params, world, ms_step), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"{name} AdamW, AL8 second moment (block {args.v_block}) + UF8 "
                               f"momentum (block 256)",
                   "tensors": len(tens), "params_per_gpu": n_params,
                   "bytes_per_step": nbytes,
                   "l2": "no flush: each step streams 17.7 GB (> 129 MB L2)",
                   "parallelism": f"replicas x{world}"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "frac_of_8tbs_spec": achieved / 8000.0,
                     "traffic": traffic,
                     "peak_source": f"{peak_src} hbm_gbs", "kernel": "adamw_fused_kernel"},
        "cpu_baseline": cpu, "e2e": e2e, "clocks": clocks, "gpu_launches": launches,
    }
    if rows is not None:
        line["rows"] = rows
    print(json.dumps(line), flush=True)


def run_e2e(torch, B, arrs, hp, t, steps, n_params, dev, nchunks=32):
    """The same step end to end through the public API from pinned host
    memory, run as a host-offloaded optimizer would run it: parameters,
    gradients and states live in flat pinned host buffers, and every step
    moves them to the device and parameters and states back, inside the
    timed region. Two ways are timed: the kernel stepping the host buffers
    in place (the e2e figure), and copies staged through device buffers.
    Staged: every step copies
    them to the device, steps and copies parameters and states back. The tensors are stepped in `nchunks` groups
    (one AdamW plan each) pipelined over two streams, so one group's inputs
    arrive while the previous group's results leave (the host link carries
    both directions at once); each step moves exactly the bytes of a
    copy-in / step / copy-out sequence, one copy per array kind and group."""
    keys_in = ("p", "g", "m_codes", "m_absmax", "v_codes", "v_meta")
    keys_out = ("p", "m_codes", "m_absmax", "v_codes", "v_meta")
    src = [dict(a, g=a["gs"][0]) for a in arrs]

    def nbytes(x):
        return x.numel() * x.element_size()

    # flat buffers, every slice 16-byte aligned; groups of consecutive tensors
    offs = {k: [] for k in keys_in}
    size = {k: 0 for k in keys_in}
    for a in src:
        for k in keys_in:
            offs[k].append(size[k])
            size[k] += (nbytes(a[k]) + 15) // 16 * 16
    dflat = {k: torch.empty(size[k], dtype=torch.uint8, device=dev) for k in keys_in}
    hflat = {k: torch.empty(size[k], dtype=torch.uint8).pin_memory() for k in keys_in}
    views = []
    for i, a in enumerate(src):
        views.append({k: dflat[k][offs[k][i]:offs[k][i] + nbytes(a[k])].view(a[k].dtype)
                      for k in keys_in})
        for k in keys_in:
            views[i][k].copy_(a[k])
            hflat[k][offs[k][i]:offs[k][i] + nbytes(a[k])].copy_(
                views[i][k].view(torch.uint8).cpu())
    target = n_params / nchunks
    groups, cur, acc = [], [], 0
    for i, a in enumerate(src):
        cur.append(i)
        acc += a["p"].numel()
        if acc >= target * (len(groups) + 1) and len(groups) < nchunks - 1:
            groups.append(cur)
            cur = []
    if cur:
        groups.append(cur)
    plans, ranges = [], []
    for grp in groups:
        plans.append(B.AdamWPlan([dict(p=views[i]["p"], g=views[i]["g"],
                                       m_codes=views[i]["m_codes"],
                                       m_absmax=views[i]["m_absmax"],
                                       v_codes=views[i]["v_codes"],
                                       v_meta=views[i]["v_meta"]) for i in grp], 256, 256, 8))
        lo, hi = grp[0], grp[-1]
        ranges.append({k: (offs[k][lo], offs[k][hi] + nbytes(src[hi][k])) for k in keys_in})
    h2d = sum(nbytes(a[k]) for a in src for k in keys_in)
    d2h = sum(nbytes(a[k]) for a in src for k in keys_out)
    main = torch.cuda.current_stream(dev)
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    done_out = [None] * len(groups)
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    ev0.record(main)
    s_in.wait_stream(main)
    for _ in range(steps):
        t += 1
        for c, (plan, r) in enumerate(zip(plans, ranges)):
            if done_out[c] is not None:
                s_in.wait_event(done_out[c])  # the previous step's results of this group left
            with torch.cuda.stream(s_in):
                for k in keys_in:
                    dflat[k][r[k][0]:r[k][1]].copy_(hflat[k][r[k][0]:r[k][1]], non_blocking=True)
            plan.step(hp, t, stream=s_in)
            stepped = torch.cuda.Event()
            stepped.record(s_in)
            s_out.wait_event(stepped)
            with torch.cuda.stream(s_out):
                for k in keys_out:
                    hflat[k][r[k][0]:r[k][1]].copy_(dflat[k][r[k][0]:r[k][1]], non_blocking=True)
            done_out[c] = torch.cuda.Event()
            done_out[c].record(s_out)
    main.wait_stream(s_out)
    main.wait_stream(s_in)
    ev1.record(main)
    torch.cuda.synchronize(dev)
    ms_staged = ev0.elapsed_time(ev1) / steps

    # The same step with the kernel reading and writing the pinned host
    # buffers in place (their device mapping, zero-copy over the host link):
    # one plan over the whole set, one launch per step, the same bytes in and
    # out. This is the e2e figure; the staged pipeline above is reported
    # beside it.
    hplan = B.AdamWPlan([{k: hflat[k][offs[k][i]:offs[k][i] + nbytes(a[k])].view(a[k].dtype)
                          for k in keys_in} for i, a in enumerate(src)], 256, 256, 8, device=dev)
    t += 1
    hplan.step(hp, t, stream=main)
    torch.cuda.synchronize(dev)
    ev0.record(main)
    for _ in range(steps):
        t += 1
        hplan.step(hp, t, stream=main)
    ev1.record(main)
    torch.cuda.synchronize(dev)
    ms = ev0.elapsed_time(ev1) / steps
    return {"value": n_params / (ms * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": ms, "steps": steps,
            "pipeline": "one fused launch per step over flat pinned host buffers, read and "
                        "written in place by the kernel across the host link",
            "staged": {"ms_per_step": ms_staged, "value": n_params / (ms_staged * 1e-3),
                       "pipeline": f"copy engines: {len(groups)} groups of tensors, inputs "
                                   "in and results out on 2 streams, flat pinned host buffers"},
            "_steps_done": 2 * steps + 1}


# ---------------------------------------------------------- reference arm --
def run_reference(args):
    """The CPU oracle as the reference arm: each step is one oracle AdamW step
    over a bounded sample of the workload (a slice of the TinyLlama draws,
    sized from a calibration step so that warmup + steps take about 100 s,
    between 1M and 256M parameters), on this host's cores (the oracle's
    OpenMP build where the compiler has OpenMP: the same results as the
    single-threaded build)."""
    import numpy as np

    import oracle as ora
    from paper_2608_22322_gb300 import workloads as wl
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    threads = oracle_threads(ora, True)
    hp = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01,
              log_floor=float(np.float32(np.log2(1e-16))))

    def state(n):
        p = (wl.rng(1).standard_normal(n) * 0.02).astype(np.float32)
        gs = [wl.gaussian_grad((n,), 1e-3, 10 + k, wl.zero_mask((n,), 0.01, 20 + k))
              for k in range(2)]
        return (p, gs, np.zeros(n, np.int8), np.zeros(n // 256, np.float32),
                np.zeros(n, np.uint8), np.zeros(2 * n // 256, np.float32))

    n0 = 1 << 22
    p, gs, mc, ma, vc, vm = state(n0)
    t0 = time.perf_counter()
    ora.adamw_step(p, gs[1], mc, ma, vc, vm, 256, 256, 8, hp, 1)
    rate = n0 / (time.perf_counter() - t0)
    n = int(100.0 * rate / max(1, args.steps + args.warmup)) // 4096 * 4096
    n = max(1 << 20, min(1 << 28, n))
    p, gs, mc, ma, vc, vm = state(n)
    t = 0
    for _ in range(args.warmup):
        t += 1
        ora.adamw_step(p, gs[t % 2], mc, ma, vc, vm, 256, 256, 8, hp, t)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        t += 1
        ora.adamw_step(p, gs[t % 2], mc, ma, vc, vm, 256, 256, 8, hp, t)
    dt = (time.perf_counter() - t0) / args.steps
    oracle_threads(ora, False)
    v = n / dt
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT,
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": dt * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": "tinyllama-1.1b AdamW, AL8 second moment + UF8 momentum, "
                                   "blocks 256", "sample": f"{n} params per step"},
            "cpu_baseline": dict({"value": v, "unit": UNIT, "cores": threads, "kind": "oracle",
                                  "sample": f"one oracle step over {n} params per timed step "
                                            f"on {threads} thread{'s' if threads > 1 else ''}"},
                                 **host_info()),
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------- the other hot-path rows --
ROW_METRICS = {
    "adafactor": "optimizer-step params/sec and achieved HBM GB/s, Adafactor (AL16 factors, "
                 "UF8 momentum)",
    "came": "optimizer-step params/sec and achieved HBM GB/s, CAME (AL16 factored V and C, "
            "UF8 momentum)",
    "apollo": "optimizer-step params/sec and achieved HBM GB/s, APOLLO (rank-256 projection, "
              "UF8 M^P, AL8 V^P)",
    "codec": "codec elements/sec and achieved HBM GB/s, AL8 and UF8 encode + decode",
}


def _device_student_t(torch, t, scale, nu, seed):
    """scale * z / sqrt(chi2_nu / nu), drawn on the device from a seeded
    generator (nu integer: chi2 as a sum of nu squared normals)."""
    gen = torch.Generator(device=t.device)
    gen.manual_seed(seed)
    t.normal_(0.0, 1.0, generator=gen)
    chi = torch.zeros_like(t)
    z = torch.empty_like(t)
    for _ in range(int(nu)):
        z.normal_(0.0, 1.0, generator=gen)
        chi.addcmul_(z, z)
    t.mul_(scale).div_(torch.sqrt(chi / nu))
    del chi, z


def _row_adafactor(torch, np, wl, B, dev):
    """Adafactor on one 4096 x 4096 weight: row and column factors AL16 in
    blocks of 128, momentum UF8 in blocks of 256, gradients N(0, 1e-3) with a
    lognormal(0, 1) scale per column and 5% exact zeros. Algorithmic bytes:
    G read once (4), p read and written (8), momentum codes read and written
    (2), absmax and factor states; the factored sums make the library read G
    three times (22 B/param), which is not counted."""
    cfg = wl.CONFIGS["adafactor"]
    rows, cols = cfg["shape"]
    n = rows * cols
    hp = dict(lr=cfg["lr"], eps1=cfg["eps1"], clip_d=cfg["clip_d"], decay_rate=cfg["decay_rate"],
              beta1=cfg["beta1"], weight_decay=cfg["weight_decay"],
              log_floor=float(np.float32(np.log2(cfg["eps1"]))))
    p = torch.empty(n, dtype=torch.float32, device=dev)
    wl.torch_device_normal_(p, 0.02, 20262)
    colscale = torch.from_numpy(wl.rng(20263).lognormal(0.0, 1.0, cols).astype(np.float32)).to(dev)
    gs = []
    for k in range(2):
        g = torch.empty(n, dtype=torch.float32, device=dev)
        wl.torch_device_normal_(g, cfg["grad_std"], 20270 + k)
        g.view(rows, cols).mul_(colscale)
        wl.torch_device_zero_(g, cfg["zero_frac"], 20280 + k)
        gs.append(g)
    fb, fbits = cfg["fac_block"], cfg["fac_bits"]
    st = {}
    for name, m in (("r", rows), ("c", cols)):
        st[name] = (torch.zeros(m, dtype=torch.int16, device=dev),
                    torch.zeros(2 * ((m + fb - 1) // fb), dtype=torch.float32, device=dev))
    mc = torch.zeros(n, dtype=torch.int8, device=dev)
    ma = torch.zeros((n + 255) // 256, dtype=torch.float32, device=dev)
    ws = torch.empty(B.al_workspace_size(B.AL_OP_ADAFACTOR, rows, cols), dtype=torch.uint8,
                     device=dev)

    def step(t):
        B.al_adafactor_step(p, gs[t % 2], rows, cols, st["r"][0], st["r"][1], st["c"][0],
                            st["c"][1], fbits, fb, mc, ma, 256, hp, t, ws)

    fac = sum(2 * 2 * m + 16 * ((m + fb - 1) // fb) for m in (rows, cols))
    nbytes = 14 * n + 8 * ma.numel() + fac

    def oracle_sample(ora, t):
        import numpy as np_
        ph, gh = p.cpu().numpy().copy(), gs[0].cpu().numpy()
        rc, rm = st["r"][0].cpu().numpy().view(np_.uint16).copy(), st["r"][1].cpu().numpy().copy()
        cc, cm = st["c"][0].cpu().numpy().view(np_.uint16).copy(), st["c"][1].cpu().numpy().copy()
        mch, mah = mc.cpu().numpy().copy(), ma.cpu().numpy().copy()
        t0 = time.perf_counter()
        ora.adafactor_step(ph, gh, rows, cols, rc, rm, cc, cm, fbits, fb, mch, mah, 256, hp, t)
        dt = time.perf_counter() - t0
        return n / dt, f"one step of the whole {rows}x{cols} matrix ({dt:.2f} s)"

    return dict(step=step, n=n, bytes=nbytes, launches=6, oracle=oracle_sample,
                workload=f"Adafactor {rows}x{cols}, AL16 factors block 128, UF8 momentum block 256",
                bytes_note="algorithmic minimum 14.03 B/param (G read once)")


def _row_came(torch, np, wl, B, dev):
    """CAME on 22 matrices of 2048 x 5632 (253,755,392 params): factored V
    and confidence C in AL16 blocks of 128, UF8 momentum in blocks of 256,
    gradients 1e-3 * Student-t(3) with 5% exact zeros. Algorithmic bytes: G
    read once (4), p read and written (8), momentum codes read and written
    (2), absmax and the four factor states; the library's passes read G four
    times and the momentum codes twice (from L2 where a matrix's gradient
    stays there between its passes), which is not counted. Per-matrix steps
    on eight streams by default (see below)."""
    cfg = wl.CONFIGS["came"]
    rows, cols = cfg["shape"]
    nm = min(cfg["n_mats"], MATS) if MATS else cfg["n_mats"]
    n1 = rows * cols
    hp = dict(lr=cfg["lr"], beta1=cfg["beta1"], beta2=cfg["beta2"], beta3=cfg["beta3"],
              eps1=cfg["eps1"], eps2=cfg["eps2"], clip_d=cfg["clip_d"],
              weight_decay=cfg["weight_decay"],
              log_floor_v=float(np.float32(np.log2(cfg["eps1"]))),
              log_floor_c=float(np.float32(np.log2(cfg["eps2"]))))
    vb, cb = cfg["v_block"], cfg["c_block"]

    def fac(m, blk):
        return (torch.zeros(m, dtype=torch.int16, device=dev),
                torch.zeros(2 * ((m + blk - 1) // blk), dtype=torch.float32, device=dev))

    mats = []
    for i in range(nm):
        p = torch.empty(n1, dtype=torch.float32, device=dev)
        wl.torch_device_normal_(p, 0.02, 20300 + i)
        gs = []
        for k in range(2):
            g = torch.empty(n1, dtype=torch.float32, device=dev)
            _device_student_t(torch, g, cfg["grad_scale"], cfg["nu"], 20400 + 100 * k + i)
            wl.torch_device_zero_(g, cfg["zero_frac"], 20600 + 100 * k + i)
            gs.append(g)
        mats.append(dict(p=p, gs=gs, vr=fac(rows, vb), vc=fac(cols, vb), cr=fac(rows, cb),
                         cc=fac(cols, cb), mc=torch.zeros(n1, dtype=torch.int8, device=dev),
                         ma=torch.zeros((n1 + 255) // 256, dtype=torch.float32, device=dev)))
    # per-matrix steps (al_came_step: eight passes chained by programmatic
    # dependent launch) dealt over eight streams, so that one matrix's short
    # factor and scale passes overlap other matrices' streaming passes
    # (measured on one box: 1.566 ms on 2 streams, 1.515 on 3, 1.494 on 4,
    # 1.480 on 6, 1.478 on 8, 1.481 on 11, 1.498 on 22; 1.61 ms for grouped
    # steps over 4 groups on 4 streams);
    # ALQ_BENCH_CAME_SINGLE=0 times grouped steps instead (one launch per
    # pass over a group of matrices, ALQ_BENCH_GROUPS groups on
    # ALQ_BENCH_STREAMS streams; one plan per group and gradient buffer)
    single = os.environ.get("ALQ_BENCH_CAME_SINGLE", "1") == "1"
    ngroups = int(os.environ.get("ALQ_BENCH_GROUPS", "4"))
    groups = [mats[i::ngroups] for i in range(ngroups)]
    plans = [] if single else [[B.FactoredPlan(B.AL_OP_CAME, [
        dict(p=m["p"], g=m["gs"][k], rows=rows, cols=cols, vr_codes=m["vr"][0],
             vr_meta=m["vr"][1], vc_codes=m["vc"][0], vc_meta=m["vc"][1], cr_codes=m["cr"][0],
             cr_meta=m["cr"][1], cc_codes=m["cc"][0], cc_meta=m["cc"][1], m_codes=m["mc"],
             m_absmax=m["ma"]) for m in grp], 16, vb, 16, cb, 256) for grp in groups]
        for k in range(2)]
    nstreams = int(os.environ.get("ALQ_BENCH_STREAMS", "8" if single else str(ngroups)))
    streams = [torch.cuda.Stream(device=dev) for _ in range(nstreams)]
    wss = ([torch.empty(B.al_workspace_size(B.AL_OP_CAME, rows, cols), dtype=torch.uint8,
                        device=dev) for _ in range(nm)] if single else None)

    def step(t):
        main = torch.cuda.current_stream(dev)
        for st in streams:
            st.wait_stream(main)
        if single:
            for i, m in enumerate(mats):
                B.al_came_step(m["p"], m["gs"][t % 2], rows, cols, m["vr"][0], m["vr"][1],
                               m["vc"][0], m["vc"][1], 16, vb, m["cr"][0], m["cr"][1],
                               m["cc"][0], m["cc"][1], 16, cb, m["mc"], m["ma"], 256, hp, t,
                               wss[i], stream=streams[i % nstreams])
        else:
            for i, plan in enumerate(plans[t % 2]):
                plan.step(hp, t, stream=streams[i % nstreams])
        for st in streams:
            main.wait_stream(st)

    facb = sum(2 * 2 * mm + 16 * ((mm + blk - 1) // blk)
               for mm, blk in ((rows, vb), (cols, vb), (rows, cb), (cols, cb)))
    nbytes = nm * (14 * n1 + 8 * ((n1 + 255) // 256) + facb)

    def oracle_sample(ora, t):
        """One oracle step of every matrix (the whole workload)."""
        import numpy as np_
        h = lambda x: x.cpu().numpy().copy()
        u16 = lambda x: x.cpu().numpy().view(np_.uint16).copy()
        host = []
        for m in mats:
            host.append((h(m["p"]), m["gs"][0].cpu().numpy(),
                         [u16(m["vr"][0]), h(m["vr"][1]), u16(m["vc"][0]), h(m["vc"][1]), 16, vb,
                          u16(m["cr"][0]), h(m["cr"][1]), u16(m["cc"][0]), h(m["cc"][1]), 16, cb,
                          h(m["mc"]), h(m["ma"]), 256]))
        t0 = time.perf_counter()
        for ph, gh, args in host:
            ora.came_step(ph, gh, rows, cols, *args, hp, t)
        dt = time.perf_counter() - t0
        return nm * n1 / dt, f"one step of all {nm} {rows}x{cols} matrices ({dt:.2f} s)"

    sched = (f"per-matrix steps (al_came_step) on {nstreams} streams" if single else
             f"grouped steps (al_came_step_multi) over {ngroups} groups of matrices on "
             f"{nstreams} streams")
    return dict(step=step, n=nm * n1, bytes=nbytes, launches=8 * (nm if single else ngroups),
                oracle=oracle_sample, cpu_threads=True,
                workload=f"CAME {nm} x {rows}x{cols}, AL16 factored V and C block 128, "
                         f"UF8 momentum block 256, {sched}",
                bytes_note="algorithmic minimum 14.03 B/param (G read once)")


def _row_apollo(torch, np, wl, B, dev):
    """APOLLO over the 154 TinyLlama-1.1B attention/MLP matrices
    (968,884,224 params): one Gaussian rank-256 projection per matrix (bf16),
    projected moments UF8 / AL8 in blocks of 256, gradients N(0, 1e-3).
    Algorithmic bytes: G read for the projection and again for the scaled
    update (8), p read and written (8), projected states and their block
    constants (the projection converts G to bf16 in shared memory: no
    staging copy). FLOPs: 2 r s L per matrix for the projection. One grouped
    step (al_apollo_step_multi: three launches for all matrices)."""
    cfg = wl.CONFIGS["tinyllama_apollo"]
    r = cfg["rank"]
    hp = dict(lr=cfg["lr"], beta1=cfg["beta1"], beta2=cfg["beta2"], eps=cfg["eps"],
              alpha=cfg["alpha"], weight_decay=cfg["weight_decay"], norm_growth_gamma=0.0,
              log_floor=float(np.float32(np.log2(1e-16))), rank=r)
    mats, nbytes, flops, n_tot = [], 0, 0, 0
    shapes = wl.tinyllama_matrices()
    if MATS:
        shapes = shapes[:MATS]
    for i, (_, (rows, cols)) in enumerate(shapes):
        n1 = rows * cols
        s_, L = min(rows, cols), max(rows, cols)
        p = torch.empty(n1, dtype=torch.float32, device=dev)
        wl.torch_device_normal_(p, 0.02, 21000 + i)
        gs = []
        for k in range(2):
            g = torch.empty(n1, dtype=torch.float32, device=dev)
            wl.torch_device_normal_(g, cfg["grad_std"], 22000 + 1000 * k + i)
            gs.append(g)
        P = torch.empty(r * s_, dtype=torch.float32, device=dev)
        wl.torch_device_normal_(P, float(np.sqrt(1.0 / r)), 24000 + i)
        Pb = P.to(torch.bfloat16).view(torch.int16)
        del P
        npj = L * r
        mats.append(dict(p=p, gs=gs, rows=rows, cols=cols, P=Pb,
                         mc=torch.zeros(npj, dtype=torch.int8, device=dev),
                         ma=torch.zeros(npj // 256, dtype=torch.float32, device=dev),
                         vc=torch.zeros(npj, dtype=torch.uint8, device=dev),
                         vm=torch.zeros(2 * (npj // 256), dtype=torch.float32, device=dev),
                         prev=torch.zeros(1, dtype=torch.float32, device=dev)))
        nbytes += 16 * n1 + 4 * npj + 24 * (npj // 256)
        flops += 2 * r * s_ * L
        n_tot += n1
    # one grouped plan per gradient buffer (a plan binds its gradients)
    plans = [B.ApolloPlan([dict(p=m["p"], g=m["gs"][k], rows=m["rows"], cols=m["cols"],
                                proj=m["P"], m_codes=m["mc"], m_absmax=m["ma"],
                                v_codes=m["vc"], v_meta=m["vm"]) for m in mats], r, 8)
             for k in range(2)]

    def step(t):
        plans[t % 2].step(hp, t)

    def oracle_sample(ora, t):
        """One oracle step of layer 0's seven matrices (q, k, v, o, gate, up,
        down: 44M parameters), the projections in double."""
        h = lambda x: x.cpu().numpy().copy()
        host = []
        for m in mats[:7]:
            host.append((m["rows"], m["cols"], h(m["p"]), m["gs"][0].cpu().numpy(),
                         m["P"].cpu().numpy().view(np.uint16).copy(), h(m["mc"]), h(m["ma"]),
                         h(m["vc"]), h(m["vm"])))
        t0 = time.perf_counter()
        for rows, cols, ph, gh, Ph, mch, mah, vch, vmh in host:
            ora.apollo_step(ph, gh, rows, cols, Ph, mch, mah, 256, vch, vmh, 8, 256,
                            np.float32(0.0), hp, t)
        dt = time.perf_counter() - t0
        n = sum(x[0] * x[1] for x in host)
        return n / dt, (f"one step of layer 0's 7 matrices ({n} params) incl. the rank-{r} "
                        f"projections in double ({dt:.2f} s)")

    return dict(step=step, n=n_tot, bytes=nbytes, flops=flops, launches=3, cpu_threads=True,
                oracle=oracle_sample,
                workload=f"APOLLO TinyLlama-1.1B {len(mats)} matrices (one grouped step), "
                         f"rank {r}, UF8 M^P, AL8 V^P block 256",
                bytes_note="G twice, p read+write, projected states")


def _row_codec(torch, np, wl, B, dev):
    """AL8 encode + AL8 decode + UF8 encode + UF8 decode of 2^28 elements
    (blocks of 256): second-moment-like values 1e-6 * chi2_1 with 1% exact
    zeros for AL8, N(0, 1e-3) for UF8. Bytes: encode reads 4 and writes 1 per
    element, decode the reverse, plus block constants."""
    n = 1 << 28
    x = torch.empty(n, dtype=torch.float32, device=dev)
    wl.torch_device_normal_(x, 1.0, 25000)
    x.mul_(x).mul_(1e-6)
    wl.torch_device_zero_(x, 0.01, 25001)
    m = torch.empty(n, dtype=torch.float32, device=dev)
    wl.torch_device_normal_(m, 1e-3, 25002)
    vc = torch.empty(n, dtype=torch.uint8, device=dev)
    vm = torch.empty(2 * (n // 256), dtype=torch.float32, device=dev)
    mc = torch.empty(n, dtype=torch.int8, device=dev)
    ma = torch.empty(n // 256, dtype=torch.float32, device=dev)
    out = torch.empty(n, dtype=torch.float32, device=dev)
    floor = float(np.float32(np.log2(1e-16)))

    def step(t):
        B.al_encode(x, 256, 8, floor, vc, vm)
        B.al_decode(vc, vm, 256, 8, out)
        B.uf8_encode(m, 256, mc, ma)
        B.uf8_decode(mc, ma, 256, out)

    nbytes = 20 * n + 2 * (8 * (n // 256)) + 2 * (4 * (n // 256))

    def oracle_sample(ora, t):
        k = n
        xh = x[:k].cpu().numpy()
        t0 = time.perf_counter()
        codes, meta = ora.al_encode(xh, 256, 8, floor)
        ora.al_decode(codes, meta, 256, 8)
        dt = time.perf_counter() - t0
        return k / dt, f"AL8 encode + decode of {k} elements ({dt:.2f} s)"

    return dict(step=step, n=n, bytes=nbytes, launches=4, oracle=oracle_sample, cpu_threads=True,
                workload="codec 2^28 elements, AL8 encode+decode and UF8 encode+decode, block 256",
                bytes_note="20 B/element + block constants")


HOLD_HZ = 2.1e9   # cycles per second of a device-side wait (the SM clock's maximum)
HOLD_BATCH = 64   # timed row steps issued behind one device-side wait, at most
HOLD_MAX_MS = 50.0  # the longest device-side wait


class L2Flush:
    """Between timed steps: writes a buffer twice the L2's size, so that no
    step starts with the previous step's data in L2, then reads a second
    one as large, so that the lines the write left dirty are written back
    before the next step (outside its events) and the step starts with a
    clean L2."""

    def __init__(self, torch, dev):
        props = torch.cuda.get_device_properties(dev)
        l2 = int(getattr(props, "L2_cache_size", 0) or (129 << 20))
        self.buf = torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev)
        self.clean = torch.zeros(2 * l2 // 4, dtype=torch.float32, device=dev)
        self.sink = torch.empty((), dtype=torch.float32, device=dev)

    def __call__(self):
        self.buf.zero_()
        torch_sum = self.clean.sum
        self.sink.copy_(torch_sum())


def measure_row(name, args, dev, warmup, min_steps, with_cpu, summary):
    """Times one non-headline hot-path row: whole steps (all of the row's
    launches) with CUDA events around each step and an L2 flush between
    steps (outside the events), issued in batches behind a device-side wait
    so that the host's launch time never shows, at least min_steps steps
    and enough to fill
    about 0.6 s, with nvidia-smi clock samples over the timed loop; bytes
    per step over time against the measured HBM copy peak; the oracle on a
    bounded sample (its OpenMP build for the multi-matrix rows)."""
    import numpy as np
    import torch

    from paper_2608_22322_gb300 import binding as B
    from paper_2608_22322_gb300 import workloads as wl

    build = {"adafactor": _row_adafactor, "came": _row_came, "apollo": _row_apollo,
             "codec": _row_codec}[name]
    w = build(torch, np, wl, B, dev)
    flush = L2Flush(torch, dev)
    stream = torch.cuda.current_stream(dev)
    t = 0
    for _ in range(max(3, warmup)):
        t += 1
        flush()
        w["step"](t)
    # calibrate the step count to fill about 0.6 s of timed steps, and the
    # host's time to issue one timed iteration
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    ev0.record(stream)
    h0 = time.perf_counter()
    for _ in range(3):
        t += 1
        flush()
        w["step"](t)
    host_ms = (time.perf_counter() - h0) * 1e3 / 3
    ev1.record(stream)
    torch.cuda.synchronize(dev)
    est = ev0.elapsed_time(ev1) / 3
    # the default run's rows fill about 0.6 s of timed steps (enough clock
    # samples); a row timed alone (--workload) runs exactly --steps steps
    steps = (min(20000, max(min_steps, int(600.0 / max(est, 1e-3)))) if summary
             else max(1, args.steps))
    props = torch.cuda.get_device_properties(dev)
    sampler = ClockSampler(str(getattr(props, "uuid", "") or "").replace("GPU-", ""))
    sampler.start()
    time.sleep(0.3)
    pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
             for _ in range(steps)]
    torch.cuda.synchronize(dev)
    # The timed steps go in batches, each behind a device-side wait (outside
    # the events) longer than twice the host's time to issue the batch: the
    # whole batch is queued before the GPU reaches it, so the events time
    # the device alone, however slow the host is at launching short steps.
    # A batch holds at most ~400 queued commands (the launch queue must not
    # fill, or the host would block behind the wait), and the wait is twice
    # the calibrated issue time of the batch, at most HOLD_MAX_MS.
    batch = max(1, min(HOLD_BATCH, 400 // (w["launches"] + 4)))
    hold_ms = min(HOLD_MAX_MS, max(0.25, 2.0 * batch * host_ms))
    i = 0
    while i < steps:
        nb = min(batch, steps - i)
        torch.cuda._sleep(int(hold_ms * 1e-3 * HOLD_HZ))
        for a, b in pairs[i:i + nb]:
            flush()
            t += 1
            a.record(stream)
            w["step"](t)
            b.record(stream)
        i += nb
    torch.cuda.synchronize(dev)
    clocks = sampler.stop()
    ms_step = sum(a.elapsed_time(b) for a, b in pairs) / steps
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", 6800.0))
    achieved = w["bytes"] / (ms_step * 1e-3) / 1e9
    unit = "params/s" if name != "codec" else "elements/s"
    cpu = None
    if with_cpu:
        import oracle as ora
        threads = oracle_threads(ora, w.get("cpu_threads", False))
        v, sample = w["oracle"](ora, t + 1)
        oracle_threads(ora, False)
        cpu = dict({"value": v, "unit": unit, "cores": threads, "kind": "oracle",
                    "sample": f"{sample} on {threads} thread{'s' if threads > 1 else ''}"},
                   **host_info())
    roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
            "frac": achieved / peak, "frac_of_8tbs_spec": achieved / 8000.0,
            "traffic": None, "peak_source": f"{peak_src} hbm_gbs",
            "kernel": "whole step (all launches; per-kernel shares in profiles/)"}
    l2 = ("L2 flushed between timed steps, outside the events: a write of twice its "
          "size, then a read of twice its size (no dirty lines left); the steps issued "
          "in batches behind a device-side wait")
    if summary:
        out = {"workload": w["workload"], "value": w["n"] / (ms_step * 1e-3), "unit": unit,
               "ms_per_step": ms_step, "steps": steps, "warmup": max(3, warmup),
               "params_per_step": w["n"], "bytes_per_step": w["bytes"], "bytes": w["bytes_note"],
               "roofline": roof, "clocks": clocks, "gpu_launches": w["launches"] * steps,
               "l2": l2, "cpu_baseline": cpu}
        if "flops" in w:
            out["projection_tflops"] = w["flops"] / (ms_step * 1e-3) / 1e12
            out["projection_note"] = "2 r s L flop per matrix over the whole step's time"
        del w
        return out
    line = {
        "metric": ROW_METRICS[name], "value": w["n"] / (ms_step * 1e-3),
        "unit": unit, "n_gpus": 1, "steps": steps, "warmup": max(3, warmup),
        "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f32", "data": "synthetic",
        "config": {"workload": w["workload"], "params_per_gpu": w["n"],
                   "bytes_per_step": w["bytes"], "bytes": w["bytes_note"], "l2": l2,
                   "parallelism": "single GPU"},
        "roofline": roof, "cpu_baseline": cpu, "e2e": None, "clocks": clocks,
        "gpu_launches": w["launches"] * steps,
    }
    if "flops" in w:
        line["projection_tflops"] = w["flops"] / (ms_step * 1e-3) / 1e12
    return line


def run_rows(args):
    """One JSON line for a non-headline hot-path row (--workload)."""
    import torch

    from paper_2608_22322_gb300 import build_lib
    build_lib.build()
    if int(os.environ.get("RANK", "0")) != 0:
        return  # the rows are single-GPU measurements
    dev = torch.device("cuda", 0)
    line = measure_row(args.workload, args, dev, warmup=args.warmup, min_steps=args.steps,
                       with_cpu=not args.no_cpu, summary=False)
    print(json.dumps(line), flush=True)


def main():
    global MATS
    args = parse_args()
    MATS = args.mats
    if args.workload != "adamw":
        run_rows(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
