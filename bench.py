#!/usr/bin/env python3
"""Benchmark of the MDS-coded matrix-multiplication hot path on GB300.

Default workload: (32,24) coded mat-multi-vec, A 65536 x 65536 fp32 (16 GiB),
a batch of 8 vectors.  One step = the whole coded pass over one batch:
encode A into its 8 parity blocks, draw the straggler set (shifted
exponential), compute all 32 worker products, decode A X from the 24
survivors.  `value` is the step's algorithmic HBM bytes divided by the step
time (GB/s); per-kernel times, the encode+decode latency, the roofline of the
dominant kernel (the worker products) and the oracle's CPU baseline ride along
on the same JSON line.  Coded gradient descent (40000 x 8000, (20,10) codes)
is measured as a secondary workload on the same line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (launched by torch.distributed.run) every rank runs the same
workload on its own GPU (independent replicas, weak scaling, no collective on
the data path); `value` sums the ranks' bytes over the slowest rank's time.
`--impl reference` times the CPU oracle on a bounded sample of the same
workload (rank 0 only).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = ("coded matvec effective HBM GB/s (% of GB300 peak); "
          "encode+decode latency µs")
CLOCK_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
REASON_NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]


# ---- algorithmic traffic (bytes that the step must move at minimum) ---------------

def step_bytes(w: synth.Workload, L: int, m: int | None = None) -> dict:
    """Algorithmic HBM bytes of one step of a mat-multi-vec workload.

    encode: read the m x d data rows once, write (n-k) L x d parity.
    worker products: read every coded element once (m d systematic + (n-k) L d
    parity), read X, write the n L x b fp64 results.
    decode: read the k L x b surviving fp64 results, write m x b fp32."""
    m = w.m if m is None else m
    par = (w.n - w.k) * L * w.d * 4
    enc = m * w.d * 4 + par
    mv = m * w.d * 4 + par + w.d * w.b * 4 + w.n * L * w.b * 8
    dec = w.k * L * w.b * 8 + m * w.b * 4
    return {"encode": enc, "matvec": mv, "decode": dec, "step": enc + mv + dec}


def gd_iter_bytes(w: synth.GDWorkload, LA: int, LAT: int) -> int:
    """Per iteration: both coded products (all coded elements once) and decodes."""
    a = w.m * w.d * 4 + (w.n - w.k_a) * LA * w.d * 4 + w.d * 4 + w.n * LA * 8
    at = w.d * w.m * 4 + (w.n - w.k_at) * LAT * w.m * 4 + w.m * 4 + w.n * LAT * 8
    dec = w.k_a * LA * 8 + 2 * w.m * 4 + w.k_at * LAT * 8 + 2 * w.d * 4
    return a + at + dec


# ---- helpers -----------------------------------------------------------------------------

NOMINAL_HBM_GBS = 7900.0   # GB300 HBM3e, nominal


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "source": "measured",
                "bf16_tflops": float(p.get("bf16_tflops", 1900.0)),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", 1700.0))}
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                "source": "fallback"}


def recorded_traffic(kernel: str, source_file: str):
    """dram bytes per launch recorded from an ncu capture, if the kernel source
    has not changed since (profiles/traffic.txt: kernel sha256 bytes note)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    if not os.path.exists(path):
        return None
    sha = hashlib.sha256(open(source_file, "rb").read()).hexdigest()
    for line in open(path):
        parts = line.split()
        if len(parts) >= 3 and not line.startswith("#") and parts[0] == kernel:
            if parts[1] == sha:
                return float(parts[2])
    return None


class ClockSampler:
    """nvidia-smi clock / throttle-reason sampling during a timed region."""

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + CLOCK_FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.15)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self) -> dict:
        sms, maxs, watts, reasons = [], [], [], set()
        try:
            for line in open(self.path):
                f = [x.strip() for x in line.split(",")]
                if len(f) < 9:
                    continue
                try:
                    sms.append(float(f[1]))
                    maxs.append(float(f[2]))
                except ValueError:
                    continue
                try:
                    watts.append(float(f[3]))
                except ValueError:
                    pass
                for name, val in zip(REASON_NAMES, f[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
            os.unlink(self.path)
        except Exception:
            pass
        if not sms:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        out = {"sm_mhz": float(np.median(sms)), "sm_max_mhz": float(max(maxs)),
               "reasons": sorted(reasons), "samples": len(sms)}
        if watts:
            out["power_w_median"] = float(np.median(watts))
            out["power_w_max"] = float(max(watts))
        return out


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    return world, rank, local


def _reduce_device():
    """Tensors for collectives live where the process group's backend wants
    them: on the GPU for NCCL, on the host for gloo."""
    import torch.distributed as dist
    return "cpu" if dist.get_backend() == "gloo" else "cuda"


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=_reduce_device())
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def whole_job_value(bytes_per_step_per_rank: int, steps: int, ms_local: float,
                    world: int) -> tuple:
    """(value in GB/s, ms): weak scaling, every rank runs its own replica of
    the workload; the job moves world x the bytes of one replica in the time
    of the slowest rank."""
    ms = max_over_ranks(ms_local, world)
    return world * bytes_per_step_per_rank * steps / (ms * 1e-3) / 1e9, ms


# ---- CPU oracle on a bounded sample (the baseline / reference arm) ---------------------

def oracle_sample_step(w: synth.Workload, s: int, seed: int, counter: int):
    """One step of the oracle on s sampled block rows of workload w: the
    sub-problem whose k blocks are s rows each (same n, k, d, b).  Returns
    (seconds, algorithmic bytes of the sample in the GPU's units)."""
    import oracle
    P = synth.parity_coefficients(w.n, w.k).astype(np.float64)
    A_sub = synth.gaussian((w.k * s, w.d), seed).numpy()
    X = synth.gaussian((w.d, w.b), seed + 1).numpy()
    t0 = time.perf_counter()
    par = oracle.encode(w.n, w.k, A_sub, P)
    Yt = oracle.worker_outputs_f64(w.n, w.k, A_sub, par, X)
    mask, _ = oracle.draw_erasures(synth.ERASURE_SEED, counter, w.n, w.k)
    oracle.decode(w.n, w.k, w.k * s, P, mask, Yt)
    dt = time.perf_counter() - t0
    return dt, step_bytes(w, s, m=w.k * s)["step"]


def cpu_baseline(w: synth.Workload, target_s: float = 12.0) -> dict:
    import oracle
    oracle.build()
    s = 4
    dt, nb = oracle_sample_step(w, s, 77, 0)
    s = int(max(4, min(w.L, s * target_s / max(dt, 1e-3) * 0.8)))
    dt, nb = oracle_sample_step(w, s, 78, 1)
    return {"value": nb / dt / 1e9, "unit": "GB/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": "%d of %d block rows of every worker (%.1f%% of the step), one step, "
                      "%.1f s" % (s, w.L, 100.0 * s / w.L, dt),
            "small_configs": oracle_small_configs()}


def oracle_small_configs() -> dict:
    """The oracle's full step (encode, all worker products, decode) on the
    tiny and the (10,5) mat-vec configurations, on every host thread and on
    one, in ms."""
    import oracle
    threads = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    out = {"threads": threads}
    for w in (synth.TINY, synth.MATVEC):
        r = {}
        for label, t in (("all_threads_ms", threads), ("one_thread_ms", 1)):
            oracle.set_threads(t)
            dt, _ = oracle_sample_step(w, w.L, 80, 0)
            r[label] = 1e3 * dt
        out[w.name] = r
    oracle.set_threads(threads)
    return out


def run_reference(args, world, rank):
    if rank != 0:
        return
    import oracle
    oracle.build()
    w = synth.BANDWIDTH
    s = 16
    for i in range(args.warmup):
        oracle_sample_step(w, s, 90 + i, i)
    tot, nb = 0.0, 0
    for i in range(args.steps):
        dt, b = oracle_sample_step(w, s, 200 + i, args.warmup + i)
        tot += dt
        nb += b
    value = nb / tot / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "GB/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": tot / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(w),
        "cpu_baseline": {"value": value, "unit": "GB/s", "cores": oracle.num_threads(),
                         "kind": "oracle",
                         "sample": "%d of %d block rows of every worker per step" % (s, w.L)},
        "e2e": {"value": value, "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# Reduced copies of the workloads for ncu captures: same codes and batch,
# inputs still larger than L2, a few GB on the device at most.  L = 608 gives
# the 152-SM mat-vec grid exactly two rounds of 8-row units.
PROFILE = synth.Workload("coded mat-multi-vec (32,24) 14592x16384 b=8 (profiling case)",
                         m=14592, d=16384, b=8, n=32, k=24, data_device="cuda")
PROFILE_GEMM = synth.Workload("coded GEMM bf16 (16,12) 18432x8192x4096 (profiling case)",
                              m=18432, d=8192, b=0, n=16, k=12, dtype="bf16", gemm_n=4096,
                              data_device="cuda")
PROFILE_SHUFFLE = synth.ShuffleWorkload("coded shuffling n=8 q=524288 s=q/4 r=256 "
                                        "(profiling case)", n=8, q=1 << 19, s=1 << 17,
                                        r=256, transitions=3)
WORKLOADS = {"bandwidth": synth.BANDWIDTH, "profile": PROFILE,
             # the (10,5) 12000 x 10000 config as the step (about 1 GB on the
             # device): the short-code kernel forms, for ncu captures
             "smallcode": synth.MATVEC}


def config_of(w: synth.Workload) -> dict:
    return {"workload": w.name, "n": w.n, "k": w.k, "m": w.m, "d": w.d, "b": w.b,
            "L": w.L, "dtype": w.dtype,
            "step": "encode + straggler draw + all n worker products + decode",
            "l2": "inputs larger than L2 (A is 16 GiB, parity 5.7 GB); no flush needed",
            "seeds": {"data": synth.DATA_SEED, "code": synth.CODE_SEED,
                      "erasure": synth.ERASURE_SEED}}


# ---- the GPU arm ---------------------------------------------------------------------------

def run_ours(args, world, rank, local):
    import paper_1512_02673_gb300 as cm

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = WORKLOADS[args.workload]
    full = args.workload == "bandwidth"
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    L = code.L
    A, X = synth.matvec_inputs(w, device=dev)
    parity = torch.empty(((w.n - w.k) * L, w.d), device=dev)
    Yt = torch.empty((w.n * L, w.b), dtype=torch.float64, device=dev)
    Y = torch.empty((w.m, w.b), device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    nbytes = step_bytes(w, L)
    stream = torch.cuda.current_stream()

    def step(counter, ev=None):
        if ev:
            ev[0].record(stream)
        cm.encode(code, A, parity, status=status)
        if ev:
            ev[1].record(stream)
        mask, _ = cm.draw_erasures(synth.ERASURE_SEED, counter, w.n, w.k)
        cm.matvec(code, A, parity, X, Yt, status=status)
        if ev:
            ev[2].record(stream)
        cm.decode(code, Yt, mask, Y=Y, status=status)
        if ev:
            ev[3].record(stream)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t_start.record(stream)
        for i in range(args.steps):
            step(args.warmup + i, evs[i])
        t_end.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms_local = t_start.elapsed_time(t_end)
    if int(status.item()) != 0:
        raise RuntimeError("device status %d during the timed steps" % int(status.item()))
    value, ms = whole_job_value(nbytes["step"], args.steps, ms_local, world)
    per = {"encode": [], "matvec": [], "decode": []}
    for e in evs:
        per["encode"].append(e[0].elapsed_time(e[1]))
        per["matvec"].append(e[1].elapsed_time(e[2]))
        per["decode"].append(e[2].elapsed_time(e[3]))
    avg = {k: float(np.mean(v)) for k, v in per.items()}
    # per step: the encode passes, the worker products and one decode launch
    launches = (math.ceil((w.n - w.k) / 16) + 1 + 1) * args.steps

    if not full and args.workload == "smallcode":   # kernels only
        if rank == 0:
            print(json.dumps({"workload": w.name, "ms_per_step": ms / args.steps,
                              "kernels_us": {k: v * 1e3 for k, v in avg.items()}}), flush=True)
        return
    if not full:   # profiling case: kernels only, then the GEMM path once per step
        del A, parity
        torch.cuda.empty_cache()
        gm = bench_gemm(cm, dev, PROFILE_GEMM, args.steps, args.warmup, sustained=False)
        torch.cuda.empty_cache()
        shf = bench_shuffle(cm, dev, PROFILE_SHUFFLE)
        if rank == 0:
            print(json.dumps({"workload": w.name, "ms_per_step": ms / args.steps,
                              "kernels_us": {k: v * 1e3 for k, v in avg.items()},
                              "gemm": gm, "coded_shuffling": shf}), flush=True)
        return

    # end to end through the public API with host buffers: pinned X in, Y out
    Xh = X.cpu().pin_memory()
    Yh = torch.empty((w.m, w.b), pin_memory=True)
    for i in range(2):
        X.copy_(Xh, non_blocking=True)
        step(1000 + i)
        Yh.copy_(Y, non_blocking=True)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    e0.record(stream)
    for i in range(args.steps):
        X.copy_(Xh, non_blocking=True)
        step(2000 + i)
        Yh.copy_(Y, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world)

    # survivors-only mode on the same workload: the straggler set is drawn
    # first and only the k surviving blocks are computed
    so = bench_survivors_only(cm, code, A, parity, X, Yt, Y, status, w, args)
    one_call = bench_one_call(cm, code, A, parity, X, Yt, Y, status, w)

    # secondary workloads: the other rows of the hot path
    del A, parity
    torch.cuda.empty_cache()
    gd = bench_gd(cm, dev, args.steps)
    torch.cuda.empty_cache()
    gemm = bench_gemm(cm, dev, synth.GEMM, max(3, args.steps // 4), args.warmup)
    torch.cuda.empty_cache()
    mv100 = bench_repeats(cm, dev, synth.MATVEC)
    tiny = bench_repeats(cm, dev, synth.TINY, repeats=20)
    torch.cuda.empty_cache()
    shuffle = bench_shuffle(cm, dev, synth.SHUFFLE)
    torch.cuda.empty_cache()
    paper = {w.name: bench_repeats(cm, dev, w) for w in synth.PAPER_MATVEC}
    paper.update({w.name: bench_gd(cm, dev, args.steps, w) for w in synth.PAPER_GD})
    torch.cuda.empty_cache()

    peaks = measured_peaks()
    achieved = nbytes["matvec"] / (avg["matvec"] * 1e-3) / 1e9
    traffic = recorded_traffic("matvec",
                               os.path.join(ROOT, "paper_1512_02673_gb300", "csrc", "k_matvec.cu"))
    line = {
        "metric": METRIC, "value": value, "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic", "config": config_of(w),
        "pct_of_peak": 100.0 * value / world / peaks["hbm_gbs"],
        "encode_decode_latency_us": {"encode": avg["encode"] * 1e3,
                                     "decode": avg["decode"] * 1e3,
                                     "sum": (avg["encode"] + avg["decode"]) * 1e3},
        "kernels": {
            "encode": {"us": avg["encode"] * 1e3,
                       "gbs": nbytes["encode"] / (avg["encode"] * 1e-3) / 1e9},
            "matvec": {"us": avg["matvec"] * 1e3, "gbs": achieved},
            "decode": {"us": avg["decode"] * 1e3,
                       "gbs": nbytes["decode"] / (avg["decode"] * 1e-3) / 1e9},
        },
        "roofline": {"bound": "hbm", "kernel": "matvec (all n worker products)",
                     "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                     "algorithmic_bytes_per_launch": nbytes["matvec"],
                     "peak_source": peaks["source"]},
        "e2e": {"value": world * nbytes["step"] * args.steps / (e2e_ms * 1e-3) / 1e9,
                "unit": "GB/s", "h2d_bytes_per_step": w.d * w.b * 4,
                "d2h_bytes_per_step": w.m * w.b * 4},
        "gpu_launches": launches,
        "clocks": clk.summary(),
        "secondary": {"survivors_only": so, "matvec_decode_one_call": one_call,
                      "gemm": gemm, "gd": gd,
                      "matvec_100_repeats": mv100, "tiny": tiny,
                      "coded_shuffling": shuffle, "paper_shaped": paper,
                      "runtime_model": runtime_model_report(cm)},
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w)
    if rank == 0:
        print(json.dumps(line), flush=True)


def bench_survivors_only(cm, code, A, parity, X, Yt, Y, status, w, args) -> dict:
    """Worker products of the k survivors only, then decode (per step)."""
    L = code.L
    masks = [cm.draw_erasures(synth.ERASURE_SEED, 3000 + i, w.n, w.k)[0]
             for i in range(args.steps + args.warmup)]
    for i in range(args.warmup):
        cm.matvec_survivors(code, A, parity, X, masks[i], Yt=Yt, status=status)
        cm.decode(code, Yt, masks[i], Y=Y, status=status)
    torch.cuda.synchronize()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    for i in range(args.steps):
        m = masks[args.warmup + i]
        ev[i][0].record()
        cm.matvec_survivors(code, A, parity, X, m, Yt=Yt, status=status)
        ev[i][1].record()
        cm.decode(code, Yt, m, Y=Y, status=status)
        ev[i][2].record()
    torch.cuda.synchronize()
    mv = float(np.mean([e[0].elapsed_time(e[1]) for e in ev]))
    dec = float(np.mean([e[1].elapsed_time(e[2]) for e in ev]))
    read = w.k * L * w.d * 4 + w.d * w.b * 4 + w.k * L * w.b * 8
    return {"matvec_ms": mv, "decode_ms": dec, "matvec_gbs": read / (mv * 1e-3) / 1e9,
            "bytes_read": read, "status": int(status.item())}


def bench_one_call(cm, code, A, parity, X, Yt, Y, status, w, reps: int = 8) -> dict:
    """Products and decode in one call (cm_matvec_decode: the decode is a
    programmatic dependent of the products) on the headline workload, all
    workers and survivors only.  Each repeat times the same products alone
    (cm_matvec / cm_matvec_survivors) and then the one call on the same
    erasure set, so the decode's added time is a median of paired
    differences."""
    ws = torch.empty(cm.matvec_decode_workspace_bytes(code, w.b), dtype=torch.uint8,
                     device=A.device)
    masks = [cm.draw_erasures(synth.ERASURE_SEED, 5000 + i, w.n, w.k)[0] for i in range(reps + 2)]
    out = {}
    for name, only in (("all_workers", False), ("survivors_only", True)):
        def alone(m):
            if only:
                cm.matvec_survivors(code, A, parity, X, m, Yt=Yt, status=status)
            else:
                cm.matvec(code, A, parity, X, Yt, status=status)

        def fused(m):
            cm.matvec_decode(code, A, parity, X, m, only_survivors=only, Y=Y, ws=ws,
                             status=status)

        for i in range(2):
            alone(masks[i])
            fused(masks[i])
        torch.cuda.synchronize()
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(reps)]
        for i, e in enumerate(ev):
            m = masks[2 + i]
            e[0].record()
            alone(m)
            e[1].record()
            e[2].record()
            fused(m)
            e[3].record()
        torch.cuda.synchronize()
        t_alone = [e[0].elapsed_time(e[1]) for e in ev]
        t_fused = [e[2].elapsed_time(e[3]) for e in ev]
        out[name] = {"ms_per_call": float(np.median(t_fused)),
                     "products_alone_ms": float(np.median(t_alone)),
                     "decode_added_us": float(np.median(np.subtract(t_fused, t_alone))) * 1e3,
                     "repeats": reps}
    out["status"] = int(status.item())
    return out


def shuffle_bytes(st: dict, r: int) -> dict:
    """Algorithmic HBM bytes of one transition's kernels: data rows of r fp32
    words plus the int32 row programs.  encode reads every summed row once and
    writes every message row; decode reads every message row once (one
    multicast for all of I), every subtracted cached row, and writes every
    received row; commit copies every received row into its cache slot."""
    R, C, X = st["uncoded_rows"], st["coded_rows"], st["subtractions"]
    rb = 4 * r
    return {"encode": (R + C) * rb + 4 * (C + 1 + R),
            "decode": (C + X + R) * rb + 4 * (3 * R + 1 + X),
            "commit": 2 * R * rb + 4 * R}


def bench_shuffle(cm, dev, w: synth.ShuffleWorkload) -> dict:
    """Coded shuffling (Sec. IV) on the GPU: per transition the host plans
    Alg. 1 and the cache update, then encode, decode by subtraction and the
    cache commit run on the device (xor sums: exact, the same bytes as real
    sums).  Then the same transitions with the planner on the device.  Checks
    after the last transition of each that every cache slot holds its data
    row exactly."""
    peaks = measured_peaks()
    A = synth.shuffle_rows(w, dev)
    sh = cm.Shuffle(w.n, w.q, w.s, synth.SHUFFLE_PARTITION_SEED, synth.SHUFFLE_CACHE_SEED)
    sh.upload()
    caches = sh.fill(A)
    M = torch.empty((w.q, w.r), device=dev)
    Rx = torch.empty((w.q, w.r), device=dev)
    rows = {"coded": [], "uncoded": []}
    t_plan, t_up, ms = [], [], {"encode": [], "decode": [], "commit": []}
    nb = {"encode": 0, "decode": 0, "commit": 0}
    for t in range(w.transitions):
        t0 = time.perf_counter()
        st = sh.next()
        t1 = time.perf_counter()
        sh.upload()
        torch.cuda.synchronize()
        t2 = time.perf_counter()
        t_plan.append(t1 - t0)
        t_up.append(t2 - t1)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        # queue the three launches behind a short device sleep, so that the
        # events time the kernels and not the host's launch gap
        torch.cuda._sleep(2_000_000)
        ev[0].record()
        sh.encode("xor", A, M)
        ev[1].record()
        sh.decode("xor", M, caches, w.r, Rx)
        ev[2].record()
        sh.commit(Rx, caches, w.r)
        ev[3].record()
        torch.cuda.synchronize()
        if t > 0:      # the first transition warms the kernels up
            for j, k in enumerate(("encode", "decode", "commit")):
                ms[k].append(ev[j].elapsed_time(ev[j + 1]))
            for k, v in shuffle_bytes(st, w.r).items():
                nb[k] += v
        rows["coded"].append(st["coded_rows"])
        rows["uncoded"].append(st["uncoded_rows"])
    _, slots = sh.caches()
    exact = bool(torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().to(dev)]))
    del sh
    # the same transitions planned on the device: plan time (CUDA events on
    # the planner's stream, and wall time including the read-back of the
    # counts) and the wall time of a whole transition (plan + data plane)
    shd = cm.Shuffle(w.n, w.q, w.s, synth.SHUFFLE_PARTITION_SEED, synth.SHUFFLE_CACHE_SEED)
    shd.device_init()
    caches = shd.fill(A, caches)
    d_plan_ev, d_plan_wall, d_trans_wall = [], [], []
    for t in range(w.transitions):
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        e0.record()
        shd.device_next()
        e1.record()
        t1 = time.perf_counter()
        shd.encode("xor", A, M)
        shd.decode("xor", M, caches, w.r, Rx)
        shd.commit(Rx, caches, w.r)
        torch.cuda.synchronize()
        t2 = time.perf_counter()
        if t > 0:
            d_plan_ev.append(e0.elapsed_time(e1))
            d_plan_wall.append(1e3 * (t1 - t0))
            d_trans_wall.append(1e3 * (t2 - t0))
    _, slots = shd.caches()
    exact_d = bool(torch.equal(caches, A[torch.from_numpy(slots.reshape(-1)).long().to(dev)]))
    rc, ru = cm.shuffle_rates(w.n, w.q, w.s)
    kern = {}
    for k in ms:
        tot = sum(ms[k])
        gbs = nb[k] / (tot * 1e-3) / 1e9
        kern[k] = {"ms": tot / len(ms[k]), "gbs": gbs, "frac": gbs / peaks["hbm_gbs"]}
    dev_ms = sum(kern[k]["ms"] for k in kern)
    return {"workload": w.name, "transitions_timed": w.transitions - 1,
            "kernels": kern, "device_ms_per_transition": dev_ms,
            "device_gbs": sum(nb.values()) / (sum(sum(v) for v in ms.values()) * 1e-3) / 1e9,
            "host_plan_ms": 1e3 * float(np.mean(t_plan[1:])),
            "upload_ms": 1e3 * float(np.mean(t_up[1:])),
            "rows": {"coded_mean": float(np.mean(rows["coded"][1:])),
                     "uncoded_mean": float(np.mean(rows["uncoded"][1:])),
                     "theorem_R_c": rc, "R_u": ru},
            "device_planner": {"plan_ms": float(np.mean(d_plan_ev)),
                               "plan_wall_ms": float(np.mean(d_plan_wall)),
                               "transition_wall_ms": float(np.mean(d_trans_wall)),
                               "caches_exact": exact_d},
            "roofline_peak_gbs": peaks["hbm_gbs"], "caches_exact": exact}


def runtime_model_report(cm) -> dict:
    """The straggler model of the paper for the bench's codes: expected overall
    runtime (units of the single-machine job) of uncoded, repetition and MDS
    schemes, the simulated MDS mean over the bench's draws, and the optimal k."""
    out = {}
    for name, n, k in [("(32,24)", 32, 24), ("(10,5)", 10, 5), ("(20,10)", 20, 10),
                       ("(16,12)", 16, 12), ("(25,23)", 25, 23), ("(10,8)", 10, 8)]:
        r = {"uncoded": cm.runtime_mean("uncoded", n, n),
             "mds": cm.runtime_mean("mds", n, k)}
        if n % k == 0:
            r["repetition"] = cm.runtime_mean("repetition", n, k)
        sim = cm.runtime_simulate("mds", n, k, 100000, seed=synth.ERASURE_SEED)
        r["mds_simulated_mean"] = float(sim.mean())
        r["mds_simulated_p95"] = float(np.percentile(sim, 95))
        ks, g = cm.optimal_mds_k(n, 1.0)
        r["k_star"], r["gamma_star"] = ks, g
        r["uncoded_over_mds"] = r["uncoded"] / r["mds"]
        out[name] = r
    return out


def bench_gd(cm, dev, steps: int, w: synth.GDWorkload = synth.GD) -> dict:
    """Coded GD (default: the 40000 x 8000 regression): seconds per iteration
    (4 launches: two coded products, two decodes with the residual and the
    descent fused into them, each a programmatic dependent of its products),
    effective GB/s over all n workers' bytes; and the survivors-only step."""
    A, _, y = synth.regression_inputs(w, device=dev)
    AT = A.t().contiguous()
    cA = cm.Code(w.n, w.k_a, w.m, w.d, synth.parity_coefficients(w.n, w.k_a))
    cAT = cm.Code(w.n, w.k_at, w.d, w.m,
                  synth.parity_coefficients(w.n, w.k_at, seed=synth.CODE_SEED + 1))
    PA = cm.encode(cA, A)
    PAT = cm.encode(cAT, AT)
    x = torch.zeros(w.d, device=dev)
    ws = torch.empty(cm.gd_workspace_bytes(cA, cAT), dtype=torch.uint8, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    masks = [(cm.draw_erasures(synth.ERASURE_SEED, 2 * t, w.n, w.k_a)[0],
              cm.draw_erasures(synth.ERASURE_SEED, 2 * t + 1, w.n, w.k_at)[0])
             for t in range(w.iters)]
    def run(survivors_only):
        x.zero_()
        for t in range(3):
            cm.gd_step(cA, A, PA, cAT, AT, PAT, y, x, w.eta, masks[t][0], masks[t][1], ws,
                       status, survivors_only=survivors_only)
        x.zero_()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        # keep the device queue ahead of the host, so that the events time the
        # iterations' kernels; the host's own enqueue time is reported beside
        torch.cuda._sleep(int(2e6 + w.iters * 1e5))
        e0.record()
        h0 = time.perf_counter()
        for t in range(w.iters):
            cm.gd_step(cA, A, PA, cAT, AT, PAT, y, x, w.eta, masks[t][0], masks[t][1], ws,
                       status, survivors_only=survivors_only)
        h1 = time.perf_counter()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / w.iters, (h1 - h0) * 1e3 / w.iters

    ms_surv, host_surv = run(True)
    x_surv = x.clone()
    ms, host = run(False)
    nb = gd_iter_bytes(w, cA.L, cAT.L)
    # the same 50 iterations as plain (uncoded) fp64 gradient descent on the
    # device: the coded iterate must follow it (Sec. III-E: decoding is exact)
    A64, y64 = A.double(), y.double()
    x64 = torch.zeros(w.d, dtype=torch.float64, device=dev)
    for t in range(w.iters):
        x64 -= w.eta * (A64.t() @ (A64 @ x64 - y64))
    rel = float(torch.linalg.norm(x.double() - x64) / torch.linalg.norm(x64))
    rel_surv = float(torch.linalg.norm(x_surv.double() - x64) / torch.linalg.norm(x64))
    del A64
    return {"workload": w.name, "iters": w.iters, "ms_per_iter": ms,
            "gbs": nb / (ms * 1e-3) / 1e9, "launches_per_iter": 4,
            "host_enqueue_ms_per_iter": host,
            "x50_rel_err_vs_fp64_gd": rel,
            "survivors_only": {"ms_per_iter": ms_surv, "host_enqueue_ms_per_iter": host_surv,
                               "x50_rel_err_vs_fp64_gd": rel_surv},
            "status": int(status.item())}


def bench_gemm(cm, dev, w: synth.Workload, steps: int, warmup: int, sustained: bool = True) -> dict:
    """Coded GEMM: bf16 encode once, then per step all n worker GEMMs on the
    tensor cores and the decode of A B from the k survivors."""
    peaks = measured_peaks()
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P, dtype="bf16")

    def flops_all(c):
        return 2.0 * w.n * c.L * w.d * w.gemm_n
    A, B = synth.gemm_inputs(w, device=dev)
    Bt = B.t().contiguous()
    del B
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    par = cm.encode(code, A)
    e1.record()
    Ct = torch.empty((w.n * code.L, w.gemm_n), device=dev)
    C = torch.empty((w.m, w.gemm_n), device=dev)
    masks = [cm.draw_erasures(synth.ERASURE_SEED, i, w.n, w.k)[0] for i in range(steps + warmup)]
    for i in range(warmup):
        cm.coded_gemm(code, A, par, Bt, Ct, status=status)
        cm.decode_mat(code, Ct, masks[i], C=C, status=status)
    torch.cuda.synchronize()
    enc_ms = e0.elapsed_time(e1)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    # keep the device queue ahead of the host (tensor maps and the cluster
    # occupancy query are prepared per call): the events time the kernels
    torch.cuda._sleep(2_000_000)
    for i in range(steps):
        ev[i][0].record()
        cm.coded_gemm(code, A, par, Bt, Ct, status=status)
        ev[i][1].record()
        cm.decode_mat(code, Ct, masks[warmup + i], C=C, status=status)
        ev[i][2].record()
    torch.cuda.synchronize()
    g_ms = float(np.mean([e[0].elapsed_time(e[1]) for e in ev]))
    g_best_ms = float(min(e[0].elapsed_time(e[1]) for e in ev))
    d_ms = float(np.mean([e[1].elapsed_time(e[2]) for e in ev]))
    # survivors only: the stragglers known before the products run, only the
    # k blocks the decode reads are computed (same masks, same decode)
    for i in range(warmup):
        cm.coded_gemm_survivors(code, A, par, Bt, masks[i], Ct, status=status)
    torch.cuda.synchronize()
    torch.cuda._sleep(2_000_000)
    for i in range(steps):
        ev[i][0].record()
        cm.coded_gemm_survivors(code, A, par, Bt, masks[warmup + i], Ct, status=status)
        ev[i][1].record()
        cm.decode_mat(code, Ct, masks[warmup + i], C=C, status=status)
        ev[i][2].record()
    torch.cuda.synchronize()
    gs_ms = float(np.mean([e[0].elapsed_time(e[1]) for e in ev]))
    ds_ms = float(np.mean([e[1].elapsed_time(e[2]) for e in ev]))
    # sustained: back to back for about 0.6 s with SM clock, power and
    # throttle reasons sampled, against the sustained (power-capped) peak
    sus = None
    if sustained:
        n_sus = max(1, int(600.0 / g_ms))
        torch.cuda.synchronize()
        with ClockSampler(torch.cuda.current_device()) as clk:
            e0.record()
            for _ in range(n_sus):
                cm.coded_gemm(code, A, par, Bt, Ct, status=status)
            e1.record()
            torch.cuda.synchronize()
        sus_ms = e0.elapsed_time(e1) / n_sus
        sus = {"gemms": n_sus, "gemm_ms": sus_ms, "tflops": flops_all(code) / (sus_ms * 1e-3) / 1e12,
               "frac_of_sustained_peak": flops_all(code) / (sus_ms * 1e-3) / 1e12
               / peaks["bf16_tflops_sustained"],
               "clocks": clk.summary()}
    flops = flops_all(code)                              # every coded row
    useful = 2.0 * w.m * w.d * w.gemm_n                  # A B itself
    tflops = flops / (g_ms * 1e-3) / 1e12
    dec_bytes = w.k * code.L * w.gemm_n * 4 + w.m * w.gemm_n * 4
    return {"workload": w.name, "steps": steps, "gemm_ms": g_ms, "tflops": tflops,
            "useful_tflops_per_step": useful / ((g_ms + d_ms) * 1e-3) / 1e12,
            "roofline": {"bound": "tensor", "kernel": "coded GEMM (tcgen05, bf16 -> fp32)",
                         "achieved": tflops, "peak": peaks["bf16_tflops"], "unit": "TFLOP/s",
                         "frac": tflops / peaks["bf16_tflops"],
                         "frac_of_sustained": tflops / peaks["bf16_tflops_sustained"],
                         # the burst peak is the best of ten cuBLAS launches:
                         # the same statistic over these steps
                         "achieved_best_of_steps": flops / (g_best_ms * 1e-3) / 1e12,
                         "frac_best_of_steps": flops / (g_best_ms * 1e-3) / 1e12
                         / peaks["bf16_tflops"],
                         "peak_source": peaks["source"] + " bf16 burst"},
            "decode_mat_ms": d_ms, "decode_mat_gbs": dec_bytes / (d_ms * 1e-3) / 1e9,
            "survivors_only": {"gemm_ms": gs_ms, "decode_mat_ms": ds_ms,
                               "tflops": 2.0 * w.k * code.L * w.d * w.gemm_n / (gs_ms * 1e-3) / 1e12,
                               "useful_tflops_per_step": useful / ((gs_ms + ds_ms) * 1e-3) / 1e12},
            "sustained": sus,
            "encode_bf16_ms": enc_ms, "status": int(status.item())}


def bench_repeats(cm, dev, w: synth.Workload, repeats: int | None = None) -> dict:
    """The paper-shaped repeat loop: encode once, then per repeat all n worker
    products and the decode from a fresh straggler set; per-call latencies."""
    P = synth.parity_coefficients(w.n, w.k)
    code = cm.Code(w.n, w.k, w.m, w.d, P)
    A, X = synth.matvec_inputs(w, device=dev)
    if w.d % 4:   # rows on a 16-byte pitch (the library's layout contract)
        Ap = torch.empty((w.m, (w.d + 3) // 4 * 4), device=dev)[:, :w.d]
        Ap.copy_(A)
        A = Ap
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    parity = cm.encode(code, A)
    torch.cuda.synchronize()
    torch.cuda._sleep(1_000_000)   # the event times the kernel, not the host's call
    e0.record()
    cm.encode(code, A, parity)
    e1.record()
    # five more back to back: the kernel's rate without one call's launch
    e2, e3 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(1_000_000)
    e2.record()
    for _ in range(5):
        cm.encode(code, A, parity)
    e3.record()
    Yt = cm.matvec(code, A, parity, X, status=status)
    Y = torch.empty((w.m, w.b), device=dev)
    reps = repeats or w.repeats
    masks = [cm.draw_erasures(synth.ERASURE_SEED, r, w.n, w.k)[0] for r in range(reps)]
    for r in range(3):
        cm.matvec(code, A, parity, X, Yt, status=status)
        cm.decode(code, Yt, masks[r], Y=Y, status=status)
    torch.cuda.synchronize()
    enc_us = e0.elapsed_time(e1) * 1e3
    enc_b2b_us = e2.elapsed_time(e3) * 1e3 / 5
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(reps)]
    # inputs that fit in L2 are flushed from it before every repeat (a write of
    # a buffer larger than L2, outside the timed events), then a read of a
    # second one, so that the flush's own dirty lines are written back before
    # the timed kernel rather than during it
    small = step_bytes(w, code.L)["matvec"] < (200 << 20)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev) if small else None
    clean = torch.ones(64 << 20, dtype=torch.int32, device=dev) if small else None

    def flush_l2(r):
        if flush is not None:
            flush.fill_(r & 255)
            clean.sum()

    # keep the device queue ahead of the host: the per-call events then time
    # the kernels, not the host's launch gaps
    torch.cuda._sleep(int(2e6 + reps * 4e5))
    for r in range(reps):
        flush_l2(r)
        ev[r][0].record()
        cm.matvec(code, A, parity, X, Yt, status=status)
        ev[r][1].record()
        cm.decode(code, Yt, masks[r], Y=Y, status=status)
        ev[r][2].record()
    torch.cuda.synchronize()
    mv = np.array([e[0].elapsed_time(e[1]) * 1e3 for e in ev])
    dec = np.array([e[1].elapsed_time(e[2]) * 1e3 for e in ev])
    # products and decode in one call (the decode a programmatic dependent of
    # the products), all n workers and the k survivors only: per repeat
    ws = torch.empty(cm.matvec_decode_workspace_bytes(code, w.b), dtype=torch.uint8, device=dev)
    one_call = {}
    for name, only in (("all_workers", False), ("survivors_only", True)):
        for r in range(3):
            cm.matvec_decode(code, A, parity, X, masks[r], only_survivors=only, Y=Y, ws=ws,
                             status=status)
        torch.cuda.synchronize()
        evs = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
        torch.cuda._sleep(int(2e6 + reps * 4e5))
        for r in range(reps):
            flush_l2(r)
            evs[r][0].record()
            cm.matvec_decode(code, A, parity, X, masks[r], only_survivors=only, Y=Y, ws=ws,
                             status=status)
            evs[r][1].record()
        torch.cuda.synchronize()
        t = np.array([e[0].elapsed_time(e[1]) * 1e3 for e in evs])
        one_call[name] = {"us_median": float(np.median(t)), "us_p95": float(np.percentile(t, 95))}
    nb = step_bytes(w, code.L)
    peaks = measured_peaks()
    mv_gbs = nb["matvec"] / (np.median(mv) * 1e-6) / 1e9
    return {"workload": w.name, "repeats": reps, "l2_flushed": flush is not None,
            "matvec_decode_one_call": one_call,
            "matvec_pct_of_measured_hbm": 100.0 * mv_gbs / peaks["hbm_gbs"],
            "matvec_pct_of_nominal_hbm": 100.0 * mv_gbs / NOMINAL_HBM_GBS,
            "encode_us": enc_us,
            "encode_gbs": nb["encode"] / (enc_us * 1e-6) / 1e9,
            "encode_us_back_to_back": enc_b2b_us,
            "encode_gbs_back_to_back": nb["encode"] / (enc_b2b_us * 1e-6) / 1e9,
            "matvec_us_median": float(np.median(mv)), "matvec_us_p95": float(np.percentile(mv, 95)),
            "matvec_gbs_median": nb["matvec"] / (np.median(mv) * 1e-6) / 1e9,
            "decode_us_median": float(np.median(dec)), "decode_us_p95": float(np.percentile(dec, 95)),
            "status": int(status.item())}


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=40)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["bandwidth", "profile", "smallcode"],
                    default="bandwidth",
                    help="profile: a 1.3 GB case of the same path, for ncu captures; "
                         "smallcode: the (10,5) 12000 x 10000 step (short-code kernels)")
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="skip the oracle timing on the host cores")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        world = int(os.environ.get("WORLD_SIZE", "1"))
        rank = int(os.environ.get("RANK", "0"))
        run_reference(args, world, rank)
        return
    world, rank, local = dist_setup()
    try:
        run_ours(args, world, rank, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
