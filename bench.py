"""Benchmark of the DNF attention forward on GB300.

Default workload: the stability stress case, bf16 SDPA forward, B=1, H=16, N_q=N_k=32768,
d_k=d_v=128, Q/K drawn 8*N(0,1) with 8 planted one-hot rows per head, V ~ N(0,1),
scale=1/sqrt(d_k), no mask: the largest single-GPU workload, and the paper's long-context length
(Section 6.2).  One step = one attention forward over that batch (the whole hot path: one kernel
launch).  `--workload 2` selects the small d=64 case, 3 and 4 the other bf16 shapes, 1 the fp32 one.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference|classical]
                    [--workload ID] [--shape B,H,N_q,N_k,d_k,d_v] [--pass fwd|bwd|qkv]
                    [--scaling weak|strong]

Prints ONE JSON line (rank 0).  `value` is whole-job TFLOP/s: FLOPs of every step on every
rank divided by the slowest rank's summed kernel time, measured with CUDA events on the
launching stream, with L2 flushed (a 256 MiB write) before every step.  `e2e` is the same
metric through moa_attn_fwd_staged (host buffers in and out, copies inside the timed region).
`--impl reference` times the fp64 CPU oracle on the host cores instead (a bounded sample of
rows per step).  `--impl classical` times the step-by-step path whose traffic the paper's
M_classical models (Section 8.2): the score matrix, its max-shifted exponentials and the
normalised weights each materialised in device memory by eager PyTorch ops (cuBLAS GEMMs and
elementwise/reduction kernels) -- a measurement of the comparison, not part of the library.
`--shape` replaces the workload's sizes (bf16, same generator) for traffic sweeps.  `--pass bwd`
times the backward pass (default workload 2) instead of the forward pass, and `--pass qkv` the
fused projection moa_qkv_proj producing that workload's Q, K, V from an input X [B, N, H*d_k].

Multi-GPU (torchrun), forward pass: the (b, h) slices of the job are independent problems and
are partitioned into contiguous ranges, one per rank; each rank runs the forward on its own
range only, and no collective touches the data (one all_reduce(MAX) of the timings).  By default
(`--scaling weak`) the job on N GPUs is N seeded instances of the workload, N*B*H slices, so
every rank owns B*H of them (rank r: the instance with seed s + 1000 r).  `--scaling strong`
partitions the workload's own B*H slices instead (fixed total work).  The backward and
projection passes run the whole workload on every rank.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2606_07713_gb300 import inputs as I  # noqa: E402

METRIC = "attention fwd TFLOP/s and % of GB300 bf16 peak; DRAM bytes vs DNF minimum"
DEFAULT_WORKLOAD = 5
# The backward and projection passes default to the d=64 workload: their CPU baselines run the
# oracle on whole (b, h) slices, which at 32768 x 32768 takes minutes per slice.
DEFAULT_WORKLOAD_OTHER_PASSES = 2
PROFILES = {2: os.path.join(ROOT, "profiles", "ncu_attn_fwd_bf16_tc_b4h16n2048d64.txt"),
            3: os.path.join(ROOT, "profiles", "ncu_attn_fwd_bf16_tc_b2h32n8192d128.txt"),
            4: os.path.join(ROOT, "profiles", "ncu_attn_fwd_bf16_tc_b8h8nq1024nk4096dk128dv64.txt"),
            5: os.path.join(ROOT, "profiles", "ncu_attn_fwd_bf16_tc_b1h16n32768d128_stress.txt")}
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2606_07713_gb300", "csrc", f)
                  for f in ("attn_fwd_bf16_tc.cu", "ptx.cuh", "tc_common.cuh")]
FLUSH_BYTES = 256 << 20


def workload_desc(cfg: I.AttnConfig) -> dict:
    s = cfg.shape
    v = "U[-1,1]" if cfg.v_dist == "uniform" else "N(0,1)"
    desc = (f"{cfg.dtype} SDPA fwd, B={s.B}, H={s.H}, N_q={s.N_q}, N_k={s.N_k}, d_k={s.d_k}, "
            f"d_v={s.d_v}, Q~{cfg.q_sigma:g}*N(0,1), K~{cfg.k_sigma:g}*N(0,1), V~{v}, "
            f"scale=1/sqrt(d_k), no mask")
    if cfg.plants_per_head:
        desc += f", {cfg.plants_per_head} planted one-hot rows per head"
    return {"workload": desc, "B": s.B, "H": s.H, "N_q": s.N_q, "N_k": s.N_k, "d_k": s.d_k,
            "d_v": s.d_v, "seed": cfg.the_seed,
            "l2": f"flushed before every step ({FLUSH_BYTES >> 20} MiB write, untimed)"}


def measured_peaks() -> tuple[dict, str]:
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        return json.load(open(p)), "measured"
    except Exception:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def kernel_source_hash() -> str:
    """sha256 of the forward kernel's sources with comments and whitespace removed, so that an
    ncu summary stays tied to the code it measured and not to its comments."""
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        text = open(f).read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()


def profiled_traffic(workload: int) -> dict | None:
    """DRAM bytes read and written per launch of the forward kernel, from the committed ncu
    summary of this workload, if it was captured from the current kernel source; else None."""
    try:
        text = open(PROFILES[workload]).read()
    except (KeyError, OSError):
        return None
    m = re.search(r"kernel_source_sha256:\s*([0-9a-f]{64})", text)
    rd = re.search(r"dram_read_bytes_per_launch:\s*([0-9.eE+]+)", text)
    wr = re.search(r"dram_write_bytes_per_launch:\s*([0-9.eE+]+)", text)
    if not m or not rd or not wr or m.group(1) != kernel_source_hash():
        return None
    return {"read": float(rd.group(1)), "write": float(wr.group(1))}


def traffic_fields(tr: dict | None, dnf: float, o_bytes: float) -> dict:
    """roofline keys from a profile's DRAM bytes.  `traffic` is ncu's read + write of one launch.
    A launch can end with part of O still dirty in L2 (written back after the kernel), which
    would make read + write fall below the DNF minimum; `traffic_vs_dnf` therefore counts the
    writes as at least |O|: (read + max(write, |O|)) / DNF."""
    if tr is None:
        return {"traffic": None, "dram_read": None, "dram_write": None, "traffic_vs_dnf": None}
    return {"traffic": tr["read"] + tr["write"], "dram_read": tr["read"], "dram_write": tr["write"],
            "traffic_vs_dnf": round((tr["read"] + max(tr["write"], o_bytes)) / dnf, 4)}


class ClockSampler:
    """nvidia-smi clock/throttle sampling every 20 ms while the timed loops run.  Each sample
    carries nvidia-smi's own timestamp; mark() records the host-clock windows of the timed loops,
    and the reported clock statistics use only the samples inside those windows."""

    QUERY = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    PERIOD_MS = 20
    REASONS = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines: list[str] = []
        self.thread = None
        self.windows: list[tuple[float, float]] = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", str(self.PERIOD_MS)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def mark(self, t0: float, t1: float) -> None:
        """A timed window, in time.time() seconds (the host's wall clock)."""
        self.windows.append((t0, t1))

    @staticmethod
    def parse(lines, windows, reasons=REASONS) -> dict:
        """Clock statistics from sample lines (see QUERY) restricted to the windows."""
        import datetime
        sm, smax, power, seen, total = [], [], [], set(), 0
        for ln in lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            try:
                t = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                vals = (float(f[2]), float(f[3]), float(f[4]))
            except ValueError:
                continue
            total += 1
            if windows and not any(a <= t <= b for a, b in windows):
                continue
            sm.append(vals[0])
            smax.append(vals[1])
            power.append(vals[2])
            for n, val in zip(reasons, f[6:10]):
                if val.lower() == "active":
                    seen.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "samples": total,
                    "samples_under_load": 0, "reasons": ["no samples inside the timed loops"]}
        return {"sm_mhz": float(np.median(sm)), "sm_min_mhz": min(sm), "sm_max_mhz": max(smax),
                "samples": total, "samples_under_load": len(sm),
                "period_ms": ClockSampler.PERIOD_MS, "power_w_max": max(power),
                "reasons": sorted(seen)}

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(2 * self.PERIOD_MS / 1000.0)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=2)
        return self.parse(self.lines, self.windows)


def reduce_max_over_ranks(values, device=None):
    """Element-wise maximum of `values` over all ranks of the default process group (identity
    when there is none): the slowest rank defines the whole job's time."""
    import torch
    import torch.distributed as dist
    t = torch.tensor(list(values), dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def whole_job_tflops(flops_per_step: float, steps: int, world: int, max_ms: float) -> float:
    """Weak scaling: every rank runs the full workload, so the job processed world * steps steps
    in the slowest rank's time."""
    return flops_per_step * steps * world / (max_ms * 1e-3) / 1e12


def job_tflops(job_flops_per_step: float, steps: int, max_ms: float) -> float:
    """TFLOP/s of a job whose steps together do job_flops_per_step (over all ranks), timed by
    the slowest rank."""
    return job_flops_per_step * steps / (max_ms * 1e-3) / 1e12


def rank_slices(scaling: str, bh: int, world: int, rank: int, seed: int):
    """(lo, hi, job_slices, seed) of this rank's part of the forward job.  The job's (b, h) slices
    are partitioned into contiguous ranges (shard.bh_range).  Weak scaling: the job is `world`
    seeded instances of the workload (world * bh slices), so rank r owns exactly instance r,
    drawn with seed + 1000 r.  Strong scaling: the job is the workload's own bh slices, split."""
    from paper_2606_07713_gb300 import shard as SH
    if scaling == "strong":
        lo, hi = SH.bh_range(bh, world, rank)
        return lo, hi, bh, seed
    lo, hi = SH.bh_range(world * bh, world, rank)
    return lo, hi, world * bh, seed + 1000 * rank


def to_device_bf16(bits, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)


# ------------------------------------------------------------------------------------------
# our arm
# ------------------------------------------------------------------------------------------
def gpu_head_start(stream) -> None:
    """Keeps the GPU busy for about a millisecond before the first timed step, so that the host
    has queued the first steps (flush, start event, kernel, end event) before the GPU reaches
    them: otherwise the host's own time to issue step 1 can fall between its two events."""
    import torch
    sleep = getattr(torch.cuda, "_sleep", None)
    if sleep is not None:
        with torch.cuda.stream(stream):
            sleep(2_000_000)


def run_ours(args, cfg: I.AttnConfig) -> None:
    import torch
    import torch.distributed as dist

    import paper_2606_07713_gb300 as pkg
    from paper_2606_07713_gb300 import shard as SH

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    pkg.lib()
    s = cfg.shape
    # This rank's (b, h) slices: a contiguous range of the job's slices (rank_slices).  A range
    # is one contiguous block of each tensor of its workload instance.
    bh_total = s.B * s.H
    strong = world > 1 and args.scaling == "strong"
    lo, hi, job_slices, seed = rank_slices(args.scaling, bh_total, world, rank, cfg.the_seed)
    x = I.make_inputs(cfg if seed == cfg.the_seed else dataclasses.replace(cfg, seed=seed))
    n_sl = hi - lo

    lo_i, hi_i = (lo, hi) if strong else (0, bh_total)   # the range inside this rank's instance
    hb = [SH.block(a, lo_i, hi_i) for a in ((x.q_bits, x.k_bits, x.v_bits) if cfg.dtype == "bf16"
                                         else (x.q, x.k, x.v))]
    if cfg.dtype == "bf16":
        hq, hk, hv = (torch.from_numpy(b.view(np.int16)).view(torch.bfloat16).pin_memory() for b in hb)
    else:
        hq, hk, hv = (torch.from_numpy(b).pin_memory() for b in hb)
    q, k, v = (t.to(dev) for t in (hq, hk, hv))
    o = torch.empty((1, n_sl, s.N_q, s.d_v), dtype=q.dtype, device=dev)
    ho = torch.empty(o.shape, dtype=o.dtype).pin_memory()
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    code = pkg.MOA_BF16 if cfg.dtype == "bf16" else pkg.MOA_FP32
    rank_flops = pkg.attn_flops(1, n_sl, s.N_q, s.N_k, s.d_k, s.d_v) if n_sl else 0.0
    flops = pkg.attn_flops(s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v)
    job_flops = flops * job_slices / bh_total
    dnf = pkg.dnf_bytes(s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v, code)
    elt = 2 if cfg.dtype == "bf16" else 4

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    def step(staged: bool):
        if n_sl == 0:
            return
        if staged:
            pkg.attn_fwd_staged(hq, hk, hv, ho, q, k, v, o, cfg.scale, stream=stream)
        else:
            pkg.attn_fwd(q, k, v, cfg.scale, out=o, stream=stream)

    # The clock sampler starts first; the warm-up steps then run right before the timed ones,
    # so that the GPU does not idle (and clock down) between them.
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.3)
    for _ in range(args.warmup):
        flush.zero_()
        step(False)
    torch.cuda.synchronize(dev)
    pkg.check(pkg.get_device_status())
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    barrier()
    t_wall = time.perf_counter()
    t0 = time.time()
    gpu_head_start(stream)
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        step(False)
        ev[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    wall = time.perf_counter() - t_wall
    kern_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = float(np.sum(kern_ms))

    # end to end: host buffers in, result back to the host, through the C ABI.  Its warm-up
    # steps (untimed) include the library's one-time creation of the staged call's streams and
    # events on this device.
    for _ in range(args.warmup):
        flush.zero_()
        step(True)
    ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    t0 = time.time()
    for i in range(args.steps):
        flush.zero_()
        ev2[i][0].record(stream)
        step(True)
        ev2[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    clocks = sampler.stop()
    e2e_step_ms = [a.elapsed_time(b) for a, b in ev2]
    e2e_ms = float(np.sum(e2e_step_ms))
    pkg.check(pkg.get_device_status())

    total_ms, e2e_ms = reduce_max_over_ranks([total_ms, e2e_ms], device=dev)

    if rank == 0:
        peaks, peak_src = measured_peaks()
        value = job_tflops(job_flops, args.steps, total_ms)
        per_launch_ms = float(np.mean(kern_ms))
        achieved = rank_flops / (per_launch_ms * 1e-3) / 1e12
        peak = float(peaks["bf16_tflops"]) if cfg.dtype == "bf16" else None
        whole_launch = n_sl == bh_total
        tr = traffic_fields(profiled_traffic(cfg.cfg_id) if whole_launch else None, dnf,
                            elt * bh_total * s.N_q * s.d_v)
        in_bytes = elt * bh_total * (s.N_q * s.d_k + s.N_k * s.d_k + s.N_k * s.d_v)
        out_bytes = elt * bh_total * s.N_q * s.d_v
        copies = job_slices / bh_total
        line = {
            "metric": METRIC,
            "value": round(value, 2),
            "unit": "TFLOP/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 6),
            "higher_is_better": True,
            "scaling": "strong" if strong else "weak",
            "vs_baseline": None,
            "dtype": cfg.dtype,
            "data": "synthetic: seeded splitmix64 + Box-Muller inputs of the workload's shape",
            "config": dict(workload_desc(cfg), parallelism=(
                "one GPU" if world == 1 else
                f"{job_slices} (b, h) slices partitioned over {world} ranks in contiguous ranges "
                f"({'the workload split' if strong else 'one seeded workload instance per rank'}; "
                f"no data collective)")),
            "pct_of_bf16_peak": round(100.0 * achieved / float(peaks["bf16_tflops"]), 2),
            "dnf_bytes": dnf,
            "roofline": {
                "bound": "tensor",
                "achieved": round(achieved, 2),
                "peak": peak,
                "peak_source": f"{peak_src} bf16_tflops (burst; kernel timed alone)",
                "unit": "TFLOP/s",
                "frac": round(achieved / peak, 4) if peak else None,
                # the same against the GEMM peak measured back to back under the power cap,
                # the other denominator for a kernel timed inside a long loop
                "frac_of_sustained": (round(achieved / float(peaks["bf16_tflops_sustained"]), 4)
                                      if peak and peaks.get("bf16_tflops_sustained") else None),
                **tr,
                "traffic_source": (os.path.relpath(PROFILES[cfg.cfg_id], ROOT)
                                   if tr["traffic"] is not None else
                                   "no ncu summary of this launch from the current kernel source"),
                "kernel": "attn_fwd_bf16_tc_kernel" if cfg.dtype == "bf16" else "attn_fwd_f32_cc_kernel",
                "achieved_from": (f"rank 0's launches over {n_sl} of {bh_total} (b, h) slices, "
                                  "CUDA events on the launching stream"),
            },
            "e2e": {
                "value": round(job_tflops(job_flops, args.steps, e2e_ms), 2),
                "unit": "TFLOP/s",
                "h2d_bytes_per_step": int(in_bytes * copies),
                "d2h_bytes_per_step": int(out_bytes * copies),
                "api": "moa_attn_fwd_staged",
                # rank 0's steps: the value above sums all of them, slow outliers included
                "ms_median": round(float(np.median(e2e_step_ms)), 6),
                "ms_max": round(float(np.max(e2e_step_ms)), 6),
            },
            # one kernel per step on every rank that owns at least one slice
            "gpu_launches": args.steps * min(world, job_slices),
            "clocks": clocks,
            "wall_s_timed_loop": round(wall, 4),
        }
        line["ms_median"] = round(float(np.median(kern_ms)), 6)
        line["ms_best"] = round(float(np.min(kern_ms)), 6)
        line["ms_max"] = round(float(np.max(kern_ms)), 6)
        if cfg.dtype == "bf16":
            sus = float(peaks.get("bf16_tflops_sustained", 1700.0))
            line["pct_of_bf16_peak_sustained"] = round(100.0 * achieved / sus, 2)
        if world == 1:
            line["cpu_baseline"] = cpu_baseline(cfg, x, budget_s=args.cpu_budget,
                                                gpu_out=o.float().reshape(-1, s.d_v))
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------------------------------
# the backward pass (--pass bwd)
# ------------------------------------------------------------------------------------------
def bwd_flops(s: I.AttnShape) -> float:
    """Algorithmic FLOPs of one backward pass: the five products S = Q K^T (rebuilt), dP = dO V^T,
    dV = W^T dO, dQ = dS K, dK = dS^T Q."""
    return 2.0 * s.B * s.H * s.N_q * s.N_k * (3 * s.d_k + 2 * s.d_v)


def bwd_bytes(s: I.AttnShape) -> float:
    """Compulsory HBM bytes of one bf16 backward pass: read Q, K, V, O, dO, LSE once, write
    dQ, dK, dV once."""
    bh = s.B * s.H
    reads = 2.0 * (s.N_q * s.d_k + s.N_k * s.d_k + s.N_k * s.d_v + 2 * s.N_q * s.d_v) + 4.0 * s.N_q
    writes = 2.0 * (s.N_q * s.d_k + s.N_k * s.d_k + s.N_k * s.d_v)
    return bh * (reads + writes)


def cpu_baseline_bwd(cfg, x, g, budget_s: float = 12.0) -> dict:
    import oracle
    orc = oracle.get()
    s = cfg.shape
    bh = s.B * s.H
    per_slice = bwd_flops(I.AttnShape(1, 1, s.N_q, s.N_k, s.d_k, s.d_v))
    q = x.q.reshape(bh, 1, s.N_q, s.d_k)
    k = x.k.reshape(bh, 1, s.N_k, s.d_k)
    v = x.v.reshape(bh, 1, s.N_k, s.d_v)
    gg = g.reshape(bh, 1, s.N_q, s.d_v)
    n = min(bh, orc.max_threads())
    t0 = time.perf_counter()
    orc.attn_bwd(q[:n], k[:n], v[:n], gg[:n], cfg.scale)
    dt = time.perf_counter() - t0
    if dt < budget_s / 4 and n < bh:
        n2 = int(min(bh, max(n, n * budget_s / max(dt, 1e-6) / 2)))
        t0 = time.perf_counter()
        orc.attn_bwd(q[:n2], k[:n2], v[:n2], gg[:n2], cfg.scale)
        dt, n = time.perf_counter() - t0, n2
    return {"value": round(per_slice * n / dt / 1e12, 6), "unit": "TFLOP/s",
            "cores": orc.max_threads(), "kind": "oracle",
            "sample": f"{n} of {bh} (b,h) slices, whole backward in fp64, {dt:.1f} s"}


def run_ours_bwd(args, cfg: I.AttnConfig) -> None:
    import torch
    import torch.distributed as dist

    import paper_2606_07713_gb300 as pkg

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    pkg.lib()
    s = cfg.shape
    if cfg.dtype != "bf16":
        raise SystemExit("the backward pass takes bf16 workloads")
    x = I.make_inputs(cfg)
    g, gbits = I.make_grad_output(cfg)
    q, k, v, do = (to_device_bf16(b, dev) for b in (x.q_bits, x.k_bits, x.v_bits, gbits))
    o, lse = pkg.attn_fwd_lse(q, k, v, cfg.scale)
    # d_k = d_v = 64: the one-kernel backward (5 tile products); otherwise the three-kernel one.
    # --bwd-path picks one explicitly.
    fused = args.bwd_path == "fused" or (args.bwd_path == "auto" and s.d_k == 64 and s.d_v == 64)
    wsb = pkg.moa_attn_bwd_fused_workspace_bytes if fused else pkg.moa_attn_bwd_workspace_bytes
    ws = torch.empty(max(16, wsb(s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v, pkg.MOA_BF16)),
                     dtype=torch.uint8, device=dev)
    host = [t.cpu().pin_memory() for t in (q, k, v, o, do, lse)]
    host_out = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in (q, k, v)]
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    flops = bwd_flops(s)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    sampler = ClockSampler(local)  # before the warm-up, as in run_ours
    sampler.start()
    time.sleep(0.3)
    for _ in range(args.warmup):
        flush.zero_()
        pkg.attn_bwd(q, k, v, o, lse, do, cfg.scale, workspace=ws, fused=fused)
    torch.cuda.synchronize(dev)
    pkg.check(pkg.get_device_status())
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    barrier()
    t0 = time.time()
    gpu_head_start(stream)
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        pkg.attn_bwd(q, k, v, o, lse, do, cfg.scale, workspace=ws, stream=stream, fused=fused)
        ev[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    kern_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = float(np.sum(kern_ms))
    # end to end: the forward's outputs and dO from pinned host memory, gradients back
    dq_, dk_, dv_ = (torch.empty_like(t) for t in (q, k, v))
    dev_in = [torch.empty_like(t) for t in (q, k, v, o, do, lse)]
    ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    t0 = time.time()
    for i in range(args.steps):
        flush.zero_()
        ev2[i][0].record(stream)
        for d_, h_ in zip(dev_in, host):
            d_.copy_(h_, non_blocking=True)
        grads = pkg.attn_bwd(*dev_in[:4], dev_in[5], dev_in[4], cfg.scale, workspace=ws,
                             stream=stream, fused=fused)
        for h_, d_ in zip(host_out, grads):
            h_.copy_(d_, non_blocking=True)
        ev2[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    clocks = sampler.stop()
    e2e_ms = float(np.sum([a.elapsed_time(b) for a, b in ev2]))
    pkg.check(pkg.get_device_status())
    total_ms, e2e_ms = reduce_max_over_ranks([total_ms, e2e_ms], device=dev)
    if rank == 0:
        peaks, peak_src = measured_peaks()
        value = whole_job_tflops(flops, args.steps, world, total_ms)
        achieved = flops / (float(np.mean(kern_ms)) * 1e-3) / 1e12
        peak = float(peaks["bf16_tflops"])
        line = {
            "metric": "attention bwd TFLOP/s (algorithmic: 5 products) and % of GB300 bf16 peak",
            "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(total_ms / args.steps, 6),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic: seeded splitmix64 + Box-Muller inputs and dO of the workload's shape",
            "config": dict(workload_desc(cfg), **{
                "workload": workload_desc(cfg)["workload"].replace("SDPA fwd", "SDPA bwd"),
                "pass": "backward (moa_attn_bwd_fused)" if fused else "backward (moa_attn_bwd)",
                "tile_products_executed_per_block_pair": 5 if fused else 7}),
            "compulsory_bytes": bwd_bytes(s),
            "roofline": {
                "bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                "peak_source": f"{peak_src} bf16_tflops (burst; call timed alone)",
                "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "traffic": None,
                "kernel": ("moa_attn_bwd_fused: attn_bwd_pre + attn_bwd_fused + attn_bwd_dq_convert"
                           if fused else
                           "moa_attn_bwd: attn_bwd_pre + attn_bwd_dkdv + attn_bwd_dq") + " (one call)",
            },
            "e2e": {
                "value": round(whole_job_tflops(flops, args.steps, world, e2e_ms), 2),
                "unit": "TFLOP/s",
                "h2d_bytes_per_step": int(sum(t.numel() * t.element_size() for t in host)),
                "d2h_bytes_per_step": int(sum(t.numel() * t.element_size() for t in host_out)),
                "api": "attn_bwd with host copies of Q, K, V, O, dO, LSE and the gradients",
            },
            "gpu_launches": 3 * args.steps,
            "clocks": clocks,
        }
        if world == 1:
            line["cpu_baseline"] = cpu_baseline_bwd(cfg, x, g, budget_s=args.cpu_budget)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ------------------------------------------------------------------------------------------
# the fused input projection (--pass qkv)
# ------------------------------------------------------------------------------------------
def proj_inputs(cfg: I.AttnConfig):
    """X [B, N, H*d_k] ~ N(0,1) and W [H*d_k, 2*H*d_k + H*d_v] ~ N(0,1)/sqrt(H*d_k) (bf16), from
    the seeded generator (streams 5 and 6), so that Q, K, V have unit scale."""
    s = cfg.shape
    dm = s.H * s.d_k
    ncol = 2 * s.H * s.d_k + s.H * s.d_v
    x64 = I.normal(cfg.the_seed, 5, s.B * s.N_q * dm)
    w64 = I.normal(cfg.the_seed, 6, dm * ncol) / math.sqrt(dm)
    xb = I.f32_to_bf16_bits(x64.astype(np.float32)).reshape(s.B, s.N_q, dm)
    wb = I.f32_to_bf16_bits(w64.astype(np.float32)).reshape(dm, ncol)
    return xb, wb


def run_ours_qkv(args, cfg: I.AttnConfig) -> None:
    import torch
    import torch.distributed as dist

    import paper_2606_07713_gb300 as pkg

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    pkg.lib()
    s = cfg.shape
    if cfg.dtype != "bf16" or s.N_q != s.N_k:
        raise SystemExit("the projection pass takes bf16 self-attention workloads (N_q = N_k)")
    xb, wb = proj_inputs(cfg)
    x, w = (to_device_bf16(b, dev) for b in (xb, wb))
    hx, hw = (torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).view(torch.bfloat16)
              .pin_memory() for b in (xb, wb))
    q = torch.empty((s.B, s.H, s.N_q, s.d_k), dtype=torch.bfloat16, device=dev)
    k = torch.empty_like(q)
    v = torch.empty((s.B, s.H, s.N_q, s.d_v), dtype=torch.bfloat16, device=dev)
    hout = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in (q, k, v)]
    flush = torch.empty(FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    dm = s.H * s.d_k
    ncol = 2 * s.H * s.d_k + s.H * s.d_v
    flops = 2.0 * s.B * s.N_q * dm * ncol

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    sampler = ClockSampler(local)  # before the warm-up, as in run_ours
    sampler.start()
    time.sleep(0.3)
    for _ in range(args.warmup):
        flush.zero_()
        pkg.qkv_proj(x, w, s.H, s.d_k, s.d_v, out=(q, k, v))
    torch.cuda.synchronize(dev)
    pkg.check(pkg.get_device_status())
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    barrier()
    t0 = time.time()
    gpu_head_start(stream)
    for i in range(args.steps):
        flush.zero_()
        ev[i][0].record(stream)
        pkg.qkv_proj(x, w, s.H, s.d_k, s.d_v, out=(q, k, v), stream=stream)
        ev[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    kern_ms = [a.elapsed_time(b) for a, b in ev]
    total_ms = float(np.sum(kern_ms))
    ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(args.steps)]
    barrier()
    t0 = time.time()
    for i in range(args.steps):
        flush.zero_()
        ev2[i][0].record(stream)
        x.copy_(hx, non_blocking=True)
        w.copy_(hw, non_blocking=True)
        pkg.qkv_proj(x, w, s.H, s.d_k, s.d_v, out=(q, k, v), stream=stream)
        for h_, d_ in zip(hout, (q, k, v)):
            h_.copy_(d_, non_blocking=True)
        ev2[i][1].record(stream)
    barrier()
    sampler.mark(t0, time.time())
    clocks = sampler.stop()
    e2e_ms = float(np.sum([a.elapsed_time(b) for a, b in ev2]))
    pkg.check(pkg.get_device_status())
    total_ms, e2e_ms = reduce_max_over_ranks([total_ms, e2e_ms], device=dev)
    if rank == 0:
        peaks, peak_src = measured_peaks()
        achieved = flops / (float(np.mean(kern_ms)) * 1e-3) / 1e12
        peak = float(peaks["bf16_tflops"])
        line = {
            "metric": "fused QKV projection TFLOP/s and % of GB300 bf16 peak",
            "value": round(whole_job_tflops(flops, args.steps, world, total_ms), 2),
            "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(total_ms / args.steps, 6), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic: seeded X ~ N(0,1), W ~ N(0,1)/sqrt(d_model)",
            "config": {"workload": f"bf16 QKV projection, X [{s.B}, {s.N_q}, {dm}] x W [{dm}, {ncol}]"
                                   f" -> Q, K [{s.B}, {s.H}, {s.N_q}, {s.d_k}], V [.., {s.d_v}]",
                       "B": s.B, "N": s.N_q, "d_model": dm, "H": s.H, "d_k": s.d_k, "d_v": s.d_v,
                       "l2": f"flushed before every step ({FLUSH_BYTES >> 20} MiB write, untimed)",
                       "pass": "projection (moa_qkv_proj)"},
            "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak,
                         "peak_source": f"{peak_src} bf16_tflops (burst; kernel timed alone)",
                         "unit": "TFLOP/s", "frac": round(achieved / peak, 4), "traffic": None,
                         "kernel": "qkv_proj_bf16_tc_kernel"},
            "e2e": {"value": round(whole_job_tflops(flops, args.steps, world, e2e_ms), 2),
                    "unit": "TFLOP/s",
                    "h2d_bytes_per_step": int(hx.numel() * 2 + hw.numel() * 2),
                    "d2h_bytes_per_step": int(sum(t.numel() * 2 for t in hout)),
                    "api": "qkv_proj with host copies of X, W and Q, K, V"},
            "gpu_launches": args.steps,
            "clocks": clocks,
        }
        if world == 1:
            line["cpu_baseline"] = cpu_baseline_qkv(cfg, xb, wb, budget_s=args.cpu_budget)
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def cpu_baseline_qkv(cfg, xb, wb, budget_s: float = 12.0) -> dict:
    import oracle
    orc = oracle.get()
    s = cfg.shape
    x = I.bf16_bits_to_f32(xb)
    w = I.bf16_bits_to_f32(wb)
    dm, ncol = w.shape
    n = min(s.N_q, 64)
    t0 = time.perf_counter()
    orc.qkv_proj(x[:1, :n], w, s.H, s.d_k, s.d_v)
    dt = time.perf_counter() - t0
    n2 = int(min(s.N_q, max(n, n * budget_s / max(dt, 1e-6) / 2)))
    t0 = time.perf_counter()
    orc.qkv_proj(x[:1, :n2], w, s.H, s.d_k, s.d_v)
    dt = time.perf_counter() - t0
    return {"value": round(2.0 * n2 * dm * ncol / dt / 1e12, 6), "unit": "TFLOP/s",
            "cores": orc.max_threads(), "kind": "oracle",
            "sample": f"{n2} of {s.B * s.N_q} tokens, fp64, {dt:.1f} s"}


# ------------------------------------------------------------------------------------------
# the classical path (what Eq. M_classical counts), for the measured traffic comparison
# ------------------------------------------------------------------------------------------
def classical_step(q, k, v, scale):
    """Eq. attention evaluated the classical way, every intermediate a device array: scaled
    scores (N_q x N_k), their row maxima, the shifted exponentials (N_q x N_k), the row sums,
    the normalised weights (N_q x N_k), then the product with V."""
    import torch
    scores = torch.matmul(q, k.transpose(-2, -1)) * scale
    shifted = scores - scores.amax(dim=-1, keepdim=True)
    expo = torch.exp(shifted)
    den = expo.sum(dim=-1, keepdim=True)
    weights = expo / den
    return torch.matmul(weights, v)


def analytic_traffic(s: I.AttnShape) -> dict:
    """Eqs. M_classical and M_MoA in elements, for N_q x N_k scores (the paper writes n for both)."""
    nn = s.N_q * s.N_k
    m_cl = s.B * s.H * (3 * nn + s.N_q * s.d_k + s.N_k * s.d_k + s.N_q + s.N_k * s.d_v)
    m_moa = s.B * s.H * (s.N_q * s.d_k + s.N_k * s.d_k + s.N_k * s.d_v)
    return {"M_classical_elements": m_cl, "M_moa_elements": m_moa,
            "k_analytic": round(m_cl / m_moa, 3)}


def run_classical(args, cfg: I.AttnConfig) -> None:
    import torch
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0 or cfg.dtype != "bf16":
        if rank == 0:
            print(json.dumps({"impl": "classical", "unavailable": "bf16 workloads only"}))
        return
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    s = cfg.shape
    x = I.make_inputs(cfg)
    q, k, v = (to_device_bf16(b, dev) for b in (x.q_bits, x.k_bits, x.v_bits))
    stream = torch.cuda.current_stream(dev)
    for _ in range(args.warmup):
        o = classical_step(q, k, v, cfg.scale)
    torch.cuda.synchronize(dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    for i in range(args.steps):
        ev[i][0].record(stream)
        o = classical_step(q, k, v, cfg.scale)
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    total_ms = float(np.sum([a.elapsed_time(b) for a, b in ev]))
    flops = 2.0 * s.B * s.H * s.N_q * s.N_k * (s.d_k + s.d_v)
    # the classical path computes the same function as the library (untimed check)
    import paper_2606_07713_gb300 as pkg
    ref = pkg.attn_fwd(q, k, v, cfg.scale).float()
    err = float((o.float() - ref).abs().max() / ref.abs().max())
    line = {
        "impl": "classical", "metric": METRIC,
        "value": round(flops * args.steps / (total_ms * 1e-3) / 1e12, 2), "unit": "TFLOP/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(total_ms / args.steps, 6), "higher_is_better": True,
        "dtype": "bf16", "data": "synthetic: seeded splitmix64 + Box-Muller inputs",
        "config": dict(workload_desc(cfg), l2="not flushed; the N_q x N_k arrays exceed L2"),
        "analytic": analytic_traffic(s),
        "dnf_bytes": 2.0 * s.B * s.H * (s.N_q * s.d_k + s.N_k * s.d_k + s.N_k * s.d_v + s.N_q * s.d_v),
        "rel_err_vs_library": err,
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------------------------
# the oracle on the host cores (cpu_baseline leg and --impl reference)
# ------------------------------------------------------------------------------------------
def _oracle_rows(cfg, x, nrows, seed):
    s = cfg.shape
    total = s.B * s.H * s.N_q
    rng = np.random.default_rng(seed)
    if nrows >= total:
        return np.arange(total, dtype=np.int64)
    return np.sort(rng.choice(total, size=nrows, replace=False)).astype(np.int64)


def _cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(cfg, x, budget_s: float = 12.0, gpu_out=None) -> dict:
    """The oracle timed on the host cores over a seeded row sample.  If the GPU output (rows of
    [B*H*N_q, d_v]) is given, the same sampled rows also give the run's parity error."""
    import oracle
    orc = oracle.get()
    s = cfg.shape
    flops_row = 2.0 * s.N_k * (s.d_k + s.d_v)
    total = s.B * s.H * s.N_q
    probe = _oracle_rows(cfg, x, min(total, 256), 1)
    t0 = time.perf_counter()
    orc.rows(x.q, x.k, x.v, cfg.scale, probe)
    dt = time.perf_counter() - t0
    n = int(min(total, max(256, len(probe) * budget_s / max(dt, 1e-6))))
    rows = _oracle_rows(cfg, x, n, 2)
    t0 = time.perf_counter()
    ref = orc.rows(x.q, x.k, x.v, cfg.scale, rows)
    dt = time.perf_counter() - t0
    out = {"value": round(flops_row * len(rows) / dt / 1e12, 6), "unit": "TFLOP/s",
           "cores": orc.max_threads(), "kind": "oracle",
           "sample": f"{len(rows)} of {total} output rows (seeded, uniform), fp64, {dt:.1f} s"}
    if gpu_out is not None:
        import torch
        got = gpu_out[torch.from_numpy(rows).to(gpu_out.device)].cpu().numpy().astype(np.float64)
        d = got - ref
        out["sampled_max_rel_err"] = float(np.max(np.abs(d)) / np.max(np.abs(ref)))
        out["sampled_rel_rms_err"] = float(np.sqrt(np.mean(d * d)) / np.sqrt(np.mean(ref * ref)))
    return out


def run_reference(args, cfg: I.AttnConfig) -> None:
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    orc = oracle.get()
    x = I.make_inputs(cfg)
    s = cfg.shape
    total = s.B * s.H * s.N_q
    flops_row = 2.0 * s.N_k * (s.d_k + s.d_v)
    # size each step's sample so the whole run stays within ~2 minutes of CPU time
    probe = _oracle_rows(cfg, x, min(total, 128), 1)
    t0 = time.perf_counter()
    orc.rows(x.q, x.k, x.v, cfg.scale, probe)
    per_row = (time.perf_counter() - t0) / len(probe)
    per_step = max(1, min(total, int(120.0 / max(1, args.steps + args.warmup) / max(per_row, 1e-9))))
    for i in range(args.warmup):
        orc.rows(x.q, x.k, x.v, cfg.scale, _oracle_rows(cfg, x, per_step, 100 + i))
    t = 0.0
    for i in range(args.steps):
        rows = _oracle_rows(cfg, x, per_step, 1000 + i)
        t0 = time.perf_counter()
        orc.rows(x.q, x.k, x.v, cfg.scale, rows)
        t += time.perf_counter() - t0
    value = flops_row * per_step * args.steps / t / 1e12
    sample = f"{per_step} of {total} output rows per step (seeded, uniform), fp64"
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s",
        "n_gpus": int(os.environ.get("WORLD_SIZE", "1")), "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(1e3 * t / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic: seeded splitmix64 + Box-Muller inputs of the workload's shape",
        "config": workload_desc(cfg),
        "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": orc.max_threads(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference", "classical"], default="ours")
    ap.add_argument("--workload", type=int, default=None, choices=sorted(I.CONFIGS),
                    help=f"workload ID (default: {DEFAULT_WORKLOAD} for the forward pass, "
                         f"{DEFAULT_WORKLOAD_OTHER_PASSES} for --pass bwd, --pass qkv and "
                         f"--impl classical)")
    ap.add_argument("--cpu-budget", type=float, default=12.0,
                    help="seconds of oracle time for the cpu_baseline sample")
    ap.add_argument("--bwd-path", choices=["auto", "fused", "split"], default="auto",
                    help="backward kernels: fused (one tile kernel, d_k = d_v = 64; its dQ is not "
                         "bitwise reproducible), split (dK/dV and dQ kernels; bitwise "
                         "reproducible), auto (fused where it applies)")
    ap.add_argument("--scaling", choices=["weak", "strong"], default="weak",
                    help="forward pass on N > 1 GPUs, slices partitioned over the ranks: weak = a "
                         "job of N workload instances (B*H slices per rank), strong = the "
                         "workload's own B*H slices split")
    ap.add_argument("--pass", dest="which", choices=["fwd", "bwd", "qkv"], default="fwd",
                    help="time the forward (default), the backward pass or the QKV projection")
    ap.add_argument("--shape", default=None,
                    help="B,H,N_q,N_k,d_k,d_v: a bf16 workload of this shape instead of --workload")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.workload is None:
        # the classical path materialises N_q x N_k arrays: 34 GB each at workload 5
        small = args.which != "fwd" or args.impl == "classical"
        args.workload = DEFAULT_WORKLOAD_OTHER_PASSES if small else DEFAULT_WORKLOAD
    cfg = I.CONFIGS[args.workload]
    if args.shape:
        dims = [int(t) for t in args.shape.split(",")]
        if len(dims) != 6 or min(dims) < 1:
            ap.error("--shape needs six positive integers B,H,N_q,N_k,d_k,d_v")
        cfg = I.custom_config(*dims, dtype="bf16", seed=sum(dims))
    if args.impl == "reference":
        run_reference(args, cfg)
    elif args.impl == "classical":
        run_classical(args, cfg)
    elif args.which == "bwd":
        run_ours_bwd(args, cfg)
    elif args.which == "qkv":
        run_ours_qkv(args, cfg)
    else:
        run_ours(args, cfg)


if __name__ == "__main__":
    main()
