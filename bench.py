#!/usr/bin/env python3
"""Benchmark of the fused M+Adam optimizer step on GB300.

One "step" is one mpadam_step over the whole tensor list (every element read
and written once).  Default workload: the LLaMA-style 7B parameter list (bf16
weights, grads and moments, stochastic rounding); the 1.5B list (E4M3
weights, fp32 moments) is measured in the same run as a secondary line.

    python bench.py [--steps K] [--warmup W] [--config llama_7b] [--impl reference]

Prints ONE JSON line (rank 0).  `value` is Gparams/s of the device-timed
step with inputs resident in HBM (all inputs are larger than L2, so no flush
is needed); `e2e` is the same metric through mpadam_step_host with pinned
host gradients in and updated weights out inside the timed region;
`roofline` relates the kernel's algorithmic bytes per launch, over its
CUDA-event duration, to the measured HBM copy bandwidth; `cpu_baseline`
times the CPU oracle on a bounded sample.  `--impl reference` times the
oracle itself as the reference arm.  Under torchrun every rank runs its own
replica of the workload (weak scaling; no collective on the data path).
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time
from datetime import datetime
from pathlib import Path

ROOT = Path(__file__).resolve().parent
sys.path.insert(0, str(ROOT))

METRIC = "fused M+Adam step Gparams/s and HBM GB/s as % of GB300 peak (1 GPU)"
UNIT = "Gparams/s"
BYTES = {"f32": 4, "bf16": 2, "e4m3": 1, "e4m3_b32": 1, "nvfp4": 0.5}


def algorithmic_bytes(wl) -> float:
    """Reads + writes of one step over the list: per element w (r+w), g (r),
    mu, nu, nu_e (r+w); per 32-element block of block-scaled E4M3 its FP16
    scale (r+w); per 16-element block of NVFP4 its E4M3 scale (r+w); per
    element of a BF16 compute copy 2 bytes (w)."""
    total = 0
    for spec, fmt in zip(wl.specs, wl.formats):
        n = spec.numel
        total += n * (2 * BYTES[fmt] + BYTES[wl.grad_dtype] + 6 * BYTES[wl.moment_dtype])
        if fmt == "e4m3_b32":
            total += 4 * ((n + 31) // 32)
        if fmt == "nvfp4":
            total += 2 * ((n + 15) // 16)
        if wl.compute_copy and fmt != "bf16":
            total += 2 * n
    return float(total)


def algorithmic_bytes_per_param(wl) -> float:
    return algorithmic_bytes(wl) / wl.n_params


# GB300's nominal HBM3e bandwidth (8 stacks at 3996 MHz), for a second fraction
# beside the measured copy peak
NOMINAL_HBM_GBS = 7900.0


def measured_peaks():
    p = ROOT / "MEASURED_PEAKS.json"
    if p.exists():
        d = json.loads(p.read_text())
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def kernel_source_hash() -> str:
    """Hash of the step kernel's sources (the files its DRAM traffic depends
    on: the kernel template, its argument layout and its instantiations),
    with comments and blank lines left out, so that editing a comment does
    not retire the recorded counters."""
    import re
    h = hashlib.sha256()
    csrc = ROOT / "paper_2607_10611_gb300" / "csrc"
    for f in sorted([csrc / "step_kernel.cuh", csrc / "step_args.h", *csrc.glob("step_*.cu")]):
        text = re.sub(r"/\*.*?\*/", "", f.read_text(), flags=re.S)
        lines = (re.sub(r"//.*$", "", ln).rstrip() for ln in text.splitlines())
        h.update("\n".join(ln for ln in lines if ln).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources (else None)."""
    p = ROOT / "profiles" / "traffic.json"
    if not p.exists():
        return None
    d = json.loads(p.read_text())
    e = d.get(workload)
    if not e or e.get("kernel_sources_sha256_16") != kernel_source_hash():
        return None
    return e.get("dram_bytes_per_launch")


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, path: Path):
        self.path = path
        self.proc = None
        try:
            self.fh = open(path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(gpu_index)], stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self, t0: float, t1: float):
        if self.proc is None or not self.path.exists():
            return None
        rows = []
        for r in csv.reader(self.path.read_text().splitlines()):
            if len(r) < 10:
                continue
            try:
                ts = datetime.strptime(r[0].strip(), "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(r[2]), float(r[3]), [x.strip() for x in r[6:10]]))
            except ValueError:
                continue
        inside = [x for x in rows if t0 - 0.05 <= x[0] <= t1 + 0.05] or rows[-3:]
        if not inside:
            return None
        mhz = sorted(x[1] for x in inside)
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for x in inside for i, v in enumerate(x[3]) if v.lower() == "active"})
        return {"sm_mhz": mhz[len(mhz) // 2], "sm_max_mhz": max(x[2] for x in inside),
                "reasons": reasons, "samples": len(inside)}


# ---------------------------------------------------------------------------
# CPU oracle timing (baseline / reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(wl, n_elems: int):
    """The first n_elems elements of the workload's tensor list, drawn on the
    host (same distributions and formats)."""
    import workloads as W
    specs, total = [], 0
    for s in wl.specs:
        if total >= n_elems:
            break
        take = min(s.numel, n_elems - total)
        specs.append(W.TensorSpec(s.name, take, s.role))
        total += take
    from dataclasses import replace
    return replace(wl, specs=tuple(specs)), total


def host_lists(mt):
    """Host numpy copies of a CPU-drawn workload for the oracle, and its FP8
    state before the first step."""
    import oracle
    import workloads as W
    tensors = [dict(w=W.to_numpy_bits(mt.w[k]), g=W.to_numpy_bits(mt.g[k]), m=W.to_numpy_bits(mt.m[k]),
                    v=W.to_numpy_bits(mt.v[k]), ve=W.to_numpy_bits(mt.ve[k])) for k in range(len(mt.w))]
    for k, b in enumerate(mt.bscale or []):
        if b is not None:
            tensors[k]["bscale"] = W.to_numpy_bits(b)
        if mt.gscale and mt.gscale[k]:
            tensors[k]["gscale"] = float(mt.gscale[k])
    fp8 = None
    if mt.fp8_exp is not None:
        fp8 = [oracle.fp8_init([tensors[k]], [mt.fp8_exp[k]])[0] if f == "e4m3" else None
               for k, f in enumerate(mt.formats)]
    return tensors, fp8


def time_oracle(wl, target_s: float, t_step: int = 1):
    """Time the oracle for one step over a sample sized for ~target_s seconds."""
    import oracle
    import workloads as W
    rate = None
    n = 1 << 18
    while True:
        swl, got = oracle_sample(wl, n)
        mt = W.materialize(swl, "cpu")
        tensors, fp8 = host_lists(mt)
        hp = oracle.hparams(stochastic=1 if wl.rounding == "stochastic" else 0, seed=wl.seed)
        kw = dict(wdt=[oracle.DTYPES[f] for f in mt.formats], gdt=oracle.DTYPES[wl.grad_dtype],
                  mdt=oracle.DTYPES[wl.moment_dtype], hp=hp, t=t_step, fp8_state=fp8)
        t0 = time.perf_counter()
        oracle.step(tensors, **kw)
        for k, x in enumerate(mt.cc or []):  # the compute copy the step also writes
            if x is not None:
                if "gscale" in tensors[k]:
                    oracle.dequant_nvfp4_bf16(tensors[k]["g"].size, tensors[k]["w"], tensors[k]["bscale"],
                                              tensors[k]["gscale"])
                elif "bscale" in tensors[k]:
                    oracle.dequant_bf16(tensors[k]["w"], bscale=tensors[k]["bscale"])
                else:
                    oracle.dequant_bf16(tensors[k]["w"], e=fp8[k][0])
        dt = time.perf_counter() - t0
        rate = got / dt
        if dt >= 0.5 * target_s or got < n:
            return got, dt, rate
        n = int(min(rate * target_s, 1 << 29))


def oracle_whole_lists(spec: str) -> dict:
    """The oracle's single-core rate on whole lists (one step each, step 1):
    ns per parameter and parameters per second."""
    import workloads as W
    out = {}
    for name in filter(None, spec.split(",")):
        wl = W.CONFIGS[name]
        got, dt, rate = time_oracle(wl, target_s=1e9)  # grows to the whole list
        out[name] = {"params": got, "whole_list": got == wl.n_params, "seconds": round(dt, 3),
                     "ns_per_param": round(1e9 / rate, 2), "gparams_per_s": rate / 1e9, "cores": 1}
    return out


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
TAIL_POOL = None  # (static share in 1/1024, chunk tiles) for mpadam_set_tail_pool, or the library's default


def run_gpu(wl, steps: int, warmup: int, rank: int, e2e_steps: int, flush_l2: bool = False):
    import torch
    import workloads as W
    from paper_2607_10611_gb300 import build

    build()
    dev = torch.device("cuda", torch.cuda.current_device())
    mt = W.materialize(wl, dev, layout="flat")
    opt = make_optimizer(wl, mt, rank)
    if TAIL_POOL:
        opt.set_tail_pool(*TAIL_POOL)
    launches_per_step = len(set(mt.formats))
    stream = torch.cuda.current_stream(dev)
    gptrs = [g.data_ptr() for g in mt.g]
    t = 1
    for _ in range(warmup):
        opt.step_ptrs(gptrs, t, stream.cuda_stream)
        t += 1
    torch.cuda.synchronize()
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    region0, region1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    # lists that fit in L2 (129 MB): between launches, outside each launch's events, a 256 MB
    # write and then a 256 MB read of another buffer, so that L2 holds none of the inputs and
    # no dirty lines whose write-back the next launch would pay for
    flush = torch.empty(64 << 20, dtype=torch.float32, device=dev) if flush_l2 else None
    flush_rd = torch.ones(64 << 20, dtype=torch.float32, device=dev) if flush_l2 else None
    if torch.distributed.is_initialized():
        torch.distributed.barrier()
    torch.cuda.synchronize()
    wall0 = time.time()
    region0.record(stream)
    for i in range(steps):
        if flush is not None:
            flush.fill_(float(i))
            flush_rd.amax()
        starts[i].record(stream)
        opt.step_ptrs(gptrs, t, stream.cuda_stream)
        ends[i].record(stream)
        t += 1
    region1.record(stream)
    torch.cuda.synchronize()
    wall1 = time.time()
    if torch.distributed.is_initialized():
        torch.distributed.barrier()
    total_ms = region0.elapsed_time(region1)
    launch_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    copy_ms = same_size_copy_ms(algorithmic_bytes(wl), flush, flush_rd, stream) if flush is not None else None
    one_tile = one_tile_step_ms(wl, rank, flush, flush_rd, stream) if flush is not None else None
    res = {"total_ms": total_ms, "launch_ms": launch_ms, "wall": (wall0, wall1),
           "grid": opt.launch_info(), "launches_per_step": launches_per_step, "l2_flushed": flush is not None,
           "copy_ms": copy_ms, "one_tile_ms": one_tile}
    del flush, flush_rd

    # end to end through the host-buffer entry point (one weight format: flat host buffers)
    if e2e_steps > 0 and "w" in mt.flat:
        # page-locked host buffers: huge-page ones from mpadam_host_buffer_alloc,
        # unless they copy clearly slower here than the driver's (torch
        # pin_memory).  A plain 1 GiB copy runs at the same rate on both, but
        # the step's chunked pipeline on the driver's buffers had steps of
        # 100-190 ms among its 87.6 ms ones (about one in five, on some boxes),
        # and none on huge pages over 40 alternating steps in one process.
        from paper_2607_10611_gb300.optimizer import HostBuffer
        probe = pinned_probe_gbs(stream)
        kinds = sorted(probe, key=lambda k: -probe[k])
        if "huge_pages" in probe and probe["huge_pages"] >= 0.95 * max(probe.values()):
            kinds = ["huge_pages"] + [k for k in kinds if k != "huge_pages"]
        nbytes = sum(x.numel() for x in mt.g) * BYTES[wl.grad_dtype] + sum(x.numel() for x in mt.w) * BYTES[wl.weight_dtype]
        for attempt, kind in enumerate(kinds):
            if kind == "huge_pages":
                hg_buf = HostBuffer(mt.flat["g"].numel(), mt.flat["g"].dtype)
                hw_buf = HostBuffer(mt.flat["w"].numel(), mt.flat["w"].dtype)
                hg, hw = hg_buf.tensor, hw_buf.tensor
            else:
                hg_buf = hw_buf = None
                hg = torch.empty(mt.flat["g"].shape, dtype=mt.flat["g"].dtype, pin_memory=True)
                hw = torch.empty(mt.flat["w"].shape, dtype=mt.flat["w"].dtype, pin_memory=True)
            # the full-size buffers can land elsewhere than the 1 GiB probe's
            # (pages on a far memory node once the near one is full): check the
            # link on them, and take the other kind if they run at under half
            # the probe's rate
            link = host_link_ms(hg, mt.flat["g"], hw, mt.flat["w"], stream)
            gbs = nbytes / (link * 1e-3) / 1e9
            if gbs >= 0.5 * probe[kind] or attempt == len(kinds) - 1:
                break
            del hg, hw
            if hg_buf is not None:
                hg_buf.free()
                hw_buf.free()
            torch.cuda.synchronize()
        res["host_buffers"] = kind
        res["host_probe_gbs"] = {k: round(v, 1) for k, v in probe.items()}
        res["host_buffers_tried"] = attempt + 1
        hg.copy_(mt.flat["g"])
        hgs = [hg[o:o + x.numel()] for o, x in zip(mt.offsets, mt.g)]
        hws = [hw[o:o + x.numel()] for o, x in zip(mt.offsets, mt.w)]
        opt.step_host(hgs, hws, t)  # warm (allocates the staging buffer)
        t += 1
        torch.cuda.synchronize()
        # one event per step boundary: the region's mean, and each step's own time
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(e2e_steps + 1)]
        ev[0].record(stream)
        for i in range(e2e_steps):
            opt.step_host(hgs, hws, t)
            ev[i + 1].record(stream)
            t += 1
        torch.cuda.synchronize()
        res["e2e_ms"] = ev[0].elapsed_time(ev[-1]) / e2e_steps
        res["e2e_step_ms"] = [ev[i].elapsed_time(ev[i + 1]) for i in range(e2e_steps)]
        res["h2d"] = sum(x.numel() for x in mt.g) * BYTES[wl.grad_dtype]
        res["d2h"] = sum(x.numel() for x in mt.w) * BYTES[wl.weight_dtype]
        res["link_ms"] = host_link_ms(hg, mt.flat["g"], hw, mt.flat["w"], stream)
        del hg, hw, hgs, hws
        if hg_buf is not None:
            hg_buf.free()
            hw_buf.free()
    opt.close()
    del mt, opt
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return res


def make_optimizer(wl, mt, rank: int):
    """The optimizer over a materialized list, as a user builds it."""
    from paper_2607_10611_gb300.optimizer import MPAdam
    extended = wl.weight_dtype not in ("bf16", "e4m3") or wl.compute_copy
    return MPAdam(mt.w, mt.m, mt.v, mt.ve, weight_dtype=mt.formats if extended else wl.weight_dtype,
                  grad_dtype=wl.grad_dtype, moment_dtype=wl.moment_dtype, rounding=wl.rounding,
                  seed=wl.seed + rank, fp8_exp=mt.fp8_exp, block_scales=mt.bscale if extended else None,
                  compute=mt.cc if extended else None, global_scales=mt.gscale if extended else None)


def one_tile_step_ms(wl, rank: int, flush, flush_rd, stream, reps: int = 20):
    """Median event-timed step over a one-tile list (3840 elements) of the
    first tensor's format, under the same flush: the launch, the kernel's
    start-up and one tile, which no list of this format can go below.
    None for lists that mix formats (two launches per step)."""
    import dataclasses
    import torch
    import workloads as W
    if len(set(wl.formats)) != 1:
        return None
    one = dataclasses.replace(wl, specs=(W.TensorSpec("one_tile", 3840, wl.specs[0].role),),
                              format_list=tuple(wl.formats[:1]) if wl.format_list else (),
                              name=wl.name + "_one_tile")
    mt = W.materialize(one, stream.device, layout="flat")
    opt = make_optimizer(one, mt, rank)
    gptrs = [g.data_ptr() for g in mt.g]
    ts = []
    for i in range(reps + 3):
        flush.fill_(float(i))
        flush_rd.amax()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        opt.step_ptrs(gptrs, i + 1, stream.cuda_stream)
        e1.record(stream)
        torch.cuda.synchronize()
        if i >= 3:
            ts.append(e0.elapsed_time(e1))
    del opt, mt
    return sorted(ts)[len(ts) // 2]


def same_size_copy_ms(nbytes: float, flush, flush_rd, stream, reps: int = 20) -> float:
    """Median event-timed device-to-device copy moving the same bytes (half
    read, half written) under the same flush: what a plain copy reaches at
    this size, where launch and DRAM latency, not bandwidth, set the time."""
    import torch
    n = max(1, int(nbytes // 2) // 4)
    a = torch.ones(n, dtype=torch.float32, device=stream.device)
    b = torch.empty_like(a)
    ts = []
    for i in range(reps):
        flush.fill_(float(i))
        flush_rd.amax()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        b.copy_(a)
        e1.record(stream)
        torch.cuda.synchronize()
        ts.append(e0.elapsed_time(e1))
    del a, b
    return sorted(ts)[len(ts) // 2]


def pinned_probe_gbs(stream) -> dict:
    """GB/s of a 1 GiB host-to-device copy from each kind of page-locked host
    buffer, best of three: 'huge_pages' (mpadam_host_buffer_alloc) and
    'driver' (torch pin_memory)."""
    import torch
    from paper_2607_10611_gb300.optimizer import HostBuffer
    n = 1 << 29
    dev = torch.empty(n, dtype=torch.bfloat16, device=stream.device)
    def best(h):
        t = float("inf")
        for _ in range(3):
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            torch.cuda.synchronize()
            a.record(stream)
            dev.copy_(h, non_blocking=True)
            b.record(stream)
            torch.cuda.synchronize()
            t = min(t, a.elapsed_time(b))
        return t
    hb = HostBuffer(n, torch.bfloat16)
    t_huge = best(hb.tensor)
    hb.free()
    hp = torch.empty(n, dtype=torch.bfloat16, pin_memory=True)
    t_drv = best(hp)
    del hp, dev
    return {"huge_pages": 2 * n / (t_huge * 1e-3) / 1e9, "driver": 2 * n / (t_drv * 1e-3) / 1e9}


def host_link_ms(h_src, d_dst, h_dst, d_src, stream, reps: int = 3) -> float:
    """The host link alone: the same bytes the end-to-end step moves (pinned
    host -> device and device -> host, concurrently on two streams), best of
    `reps`, in ms.  d_dst is rewritten with the values it already holds."""
    import torch
    up, down = torch.cuda.Stream(), torch.cuda.Stream()
    best = float("inf")
    for _ in range(reps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record(stream)
        up.wait_event(a)
        down.wait_event(a)
        with torch.cuda.stream(up):
            d_dst.copy_(h_src, non_blocking=True)
        with torch.cuda.stream(down):
            h_dst.copy_(d_src, non_blocking=True)
        stream.wait_stream(up)
        stream.wait_stream(down)
        b.record(stream)
        torch.cuda.synchronize()
        best = min(best, a.elapsed_time(b))
    return best


def run_toy(steps: int):
    """The BF16-stored matrix-fitting diagnostic: every regime with every
    update rule for `steps` steps at n = 4096, B = 65536, through
    mpadam_toy_run (graph replays).  Reports the mean device time per step
    (three kernels) and, per run, the mean loss of the last 64 steps over
    that of the first 4 (lower is better)."""
    import torch
    import workloads as W
    from paper_2607_10611_gb300.toy import ToyDiagnostic
    stream = torch.cuda.current_stream()
    out, total_ms = {}, 0.0
    for regime in W.TOY_REGIMES:
        p = W.toy_problem(regime, device="cuda", seed=0)
        out[regime] = {}
        for mode in ("additive", "multiplicative", "combined"):
            lr = W.TOY_LR[mode][regime]
            w = p.w0.clone()
            d = ToyDiagnostic(w, p.wstar, mode=mode, batch=65536, c_lo=p.c_lo, c_hi=p.c_hi, split=p.split, seed=1,
                              lr_add=lr if mode != "multiplicative" else 0.0,
                              lr_mul=lr if mode != "additive" else 0.0)
            losses = torch.zeros(steps, dtype=torch.float64, device="cuda")
            d.run(1, 64, losses[:64])           # capture the run graph (not timed)
            torch.cuda.synchronize()
            w.copy_(p.w0)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            d.run(1, steps, losses)             # CUDA-graph replays of 64 steps
            e1.record(stream)
            torch.cuda.synchronize()
            total_ms += e0.elapsed_time(e1)
            L = losses.cpu().numpy()
            out[regime][mode] = {"lr": lr, "loss_ratio": float(L[-64:].mean() / L[:4].mean()),
                                 "final_loss": float(L[-64:].mean())}
            d.close()
            del w
    return {"n": W.TOY_N, "batch": 65536, "steps_per_run": steps, "runs": 15,
            "us_per_step": 1e3 * total_ms / (15 * steps), "launches_per_step": 2, "regimes": out}


def max_over_ranks(ms: float, device: str) -> float:
    """The slowest rank's timed-region length (every rank gets it)."""
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(params_per_rank: int, ranks: int, ms_per_step: float) -> float:
    """Whole-job Gparams/s: every rank steps its own replica (weak scaling)."""
    return ranks * params_per_rank / (ms_per_step * 1e-3) / 1e9


def summarize(wl, res, n_gpus, peak, peak_kind):
    n = wl.n_params
    ms = res["total_ms"] / len(res["launch_ms"])
    if res.get("l2_flushed"):   # the region also holds the flushes: time the launches alone
        ms = res.get("launch_total_ms", sum(res["launch_ms"])) / len(res["launch_ms"])
    bpp = algorithmic_bytes_per_param(wl)
    launch = sorted(res["launch_ms"])
    avg_launch = sum(launch) / len(launch)
    achieved = algorithmic_bytes(wl) / (avg_launch * 1e-3) / 1e9
    out = {
        "workload": wl.name, "rounding": wl.rounding, "params": n, "tensors": len(wl.specs),
        "l2": "flushed between launches (256 MB write, then 256 MB read)" if res.get("l2_flushed")
              else "inputs larger than L2",
        "ms_per_step": ms, "gparams_per_s": whole_job_rate(n, n_gpus, ms),
        "hbm_gbs": algorithmic_bytes(wl) / (ms * 1e-3) / 1e9,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": recorded_traffic(wl.name),
                     "peak_source": peak_kind, "nominal_peak": NOMINAL_HBM_GBS,
                     "frac_of_nominal": round(achieved / NOMINAL_HBM_GBS, 4),
                     "bytes_per_param": round(bpp, 4),
                     "launches_per_step": res["launches_per_step"],
                     "kernel": "mpadam::step_kernel", "launch_ms_avg": round(avg_launch, 4),
                     "launch_ms_min": round(launch[0], 4), "launch_ms_max": round(launch[-1], 4)},
        "grid": res["grid"],
    }
    if res.get("copy_ms"):
        # context for lists that fit in L2: a plain copy of the same bytes, same flush
        out["roofline"]["copy_same_bytes_ms"] = round(res["copy_ms"], 4)
        out["roofline"]["frac_of_copy_same_bytes"] = round(res["copy_ms"] / avg_launch, 4)
    if res.get("one_tile_ms"):
        # the same kernel over one tile, same flush: the floor of a step of this format
        out["roofline"]["one_tile_step_ms"] = round(res["one_tile_ms"], 4)
    if "e2e_ms" in res:
        per = sorted(res["e2e_step_ms"])
        med = per[len(per) // 2] if len(per) % 2 else 0.5 * (per[len(per) // 2 - 1] + per[len(per) // 2])
        out["e2e"] = {"value": n_gpus * n / (res["e2e_ms"] * 1e-3) / 1e9, "unit": UNIT,
                      "h2d_bytes_per_step": res["h2d"], "d2h_bytes_per_step": res["d2h"],
                      "ms_per_step": round(res["e2e_ms"], 3), "steps": len(per),
                      "ms_median": round(med, 3), "ms_worst": round(per[-1], 3), "ms_best": round(per[0], 3),
                      "host_link_ms": round(res["link_ms"], 3),
                      "host_link_gbs": round((res["h2d"] + res["d2h"]) / (res["link_ms"] * 1e-3) / 1e9, 1),
                      "frac_of_host_link_bound": round(res["link_ms"] / res["e2e_ms"], 4),
                      "frac_of_host_link_bound_median": round(res["link_ms"] / med, 4),
                      "host_buffers": res.get("host_buffers"), "host_probe_gbs": res.get("host_probe_gbs"),
                      "host_buffers_tried": res.get("host_buffers_tried"),
                      "step_ms": [round(x, 3) for x in res["e2e_step_ms"]]}
    return out


def compact(sec) -> dict:
    """One secondary list in a few keys: the driver keeps only the tail of
    the line, so the full record goes to the details file."""
    c = {"workload": sec["workload"] + ("" if sec["rounding"] == W_DEFAULT_ROUNDING.get(sec["workload"]) else
                                         ":" + sec["rounding"]),
         "ms": round(sec["ms_per_step"], 4), "gparam_s": round(sec["gparams_per_s"], 1),
         "gbs": round(sec["roofline"]["achieved"], 0), "frac": sec["roofline"]["frac"]}
    if "frac_of_copy_same_bytes" in sec["roofline"]:
        c["frac_of_copy"] = sec["roofline"]["frac_of_copy_same_bytes"]
    if "one_tile_step_ms" in sec["roofline"]:
        c["one_tile_ms"] = sec["roofline"]["one_tile_step_ms"]
    clk = sec.get("clocks") or {}
    c["sm_mhz"] = clk.get("sm_mhz")
    if clk.get("reasons"):
        c["reasons"] = clk["reasons"]
    return c


W_DEFAULT_ROUNDING = {}  # workload name -> its configured rounding (filled in main)


def workload_config(wl, world: int, l2: str) -> dict:
    """The `config` of the JSON line: what the workload is (both arms print the same)."""
    return {"workload": wl.name, "params": wl.n_params, "tensors": len(wl.specs),
            "weights": wl.weight_dtype, "grads": wl.grad_dtype, "moments": wl.moment_dtype,
            "rounding": wl.rounding, "l2": l2,
            "parallelism": f"replicas x{world}" if world > 1 else "single GPU"}


def result_line(wl, world, steps, warmup, l2_desc, main_sum, cpu, clocks, toy, details, secondary,
                launches, cpu_lists=None) -> dict:
    """The one JSON line rank 0 prints.  The driver keeps only the line's
    tail, so it stays short: the full per-workload record (every roofline
    field, the diagnostic's per-regime table) is in the details file, and
    the compact secondary entries come last."""
    roof = main_sum["roofline"]
    return {
        "metric": METRIC, "value": round(main_sum["gparams_per_s"], 3), "unit": UNIT, "n_gpus": world,
        "steps": steps, "warmup": warmup, "ms_per_step": round(main_sum["ms_per_step"], 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": workload_config(wl, world, l2_desc),
        "hbm_gbs": round(main_sum["hbm_gbs"], 1),
        "roofline": {k: roof[k] for k in ("bound", "achieved", "peak", "unit", "frac", "traffic", "peak_source",
                                          "nominal_peak", "frac_of_nominal", "bytes_per_param", "launch_ms_avg")},
        "cpu_baseline": cpu,
        "cpu_ns_per_param": {k: v["ns_per_param"] for k, v in (cpu_lists or {}).items()},
        "e2e": {k: v for k, v in main_sum["e2e"].items() if k != "step_ms"} if main_sum.get("e2e") else None,
        "gpu_launches": launches,
        "grid": main_sum["grid"],
        "clocks": clocks,
        "toy_us_per_step": round(toy["us_per_step"], 2) if toy else None,
        "details": str(details),
        # last, so that the tail of the line the driver keeps holds every list
        "secondary": [compact(x) for x in secondary],
    }


def parse_secondary(spec: str):
    """'name' or 'name:rounding', comma-separated."""
    import workloads as W
    out = []
    for item in filter(None, spec.split(",")):
        name, _, rnd = item.partition(":")
        wl = W.CONFIGS[name]
        out.append(W.replace(wl, rounding=rnd) if rnd else wl)
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default="llama_7b")
    ap.add_argument("--secondary", default="llama_1p5b,llama_1p5b_mixed,llama_1p5b_nvfp4,"
                                           "llama_1p5b_nvfp4:stochastic,gpt2_124m,ragged_20k,flat_1m",
                    help="comma-separated workload[:rounding] list measured after the main one ('' to skip)")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--cpu-lists", default="flat_1m,gpt2_124m",
                    help="lists the oracle also steps whole, once each, for its single-core rate ('' skips)")
    ap.add_argument("--toy-steps", type=int, default=2048, help="matrix-fitting diagnostic steps per run (0 skips)")
    ap.add_argument("--rounding", default=None, choices=["nearest", "stochastic"],
                    help="override the workload's weight rounding")
    ap.add_argument("--clocks-dir", default=None,
                    help="directory for the raw nvidia-smi clock samples (clocks_rank0.csv) and the full "
                         "per-workload record (bench_details.json); default: the temp dir")
    ap.add_argument("--tail-pool", default=None, metavar="Q,CHUNK",
                    help="static share (1/1024) and chunk tiles of the step's tail pool (default: the library's)")
    ap.add_argument("--max-params", type=int, default=0,
                    help="truncate the list to its first N params (small profiling cases)")
    args = ap.parse_args()
    warmup = max(3, args.warmup)

    import workloads as W
    for name, w in W.CONFIGS.items():
        W_DEFAULT_ROUNDING[name] = w.rounding
    wl = W.CONFIGS[args.config]
    if args.rounding:
        wl = W.replace(wl, rounding=args.rounding)
    if args.tail_pool:
        global TAIL_POOL
        TAIL_POOL = tuple(int(x) for x in args.tail_pool.split(","))
    if args.max_params:
        wl, got = oracle_sample(wl, args.max_params)
        wl = W.replace(wl, name=f"{wl.name}[:{got}]")
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    l2_desc = ("flushed between launches (256 MB write, then 256 MB read)" if algorithmic_bytes(wl) < 512e6
               else "inputs larger than L2 (no flush needed)")

    if args.impl == "reference":
        # the oracle is the reference: rank 0 only, on the host cores
        if rank != 0:
            return
        per_step = []
        for i in range(warmup + args.steps):
            got, dt, rate = time_oracle(wl, target_s=1.0, t_step=1 + i)
            if i >= warmup:
                per_step.append((got, dt))
        elems = sum(g for g, _ in per_step)
        secs = sum(d for _, d in per_step)
        value = elems / secs / 1e9
        sample_ms = 1e3 * secs / len(per_step)
        sample = (f"each step: one oracle step over the first {per_step[-1][0]} elements of the {wl.name} list "
                  f"(single thread); ms_per_step is that sample's time")
        line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
                "steps": args.steps, "warmup": warmup, "ms_per_step": round(sample_ms, 3),
                "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                "data": "synthetic", "config": workload_config(wl, 1, l2_desc),
                "sample_elements_per_step": per_step[-1][0],
                "whole_list_ms_per_step_extrapolated": round(1e3 * wl.n_params / (value * 1e9), 1),
                "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "nproc": os.cpu_count(),
                                 "kind": "oracle", "sample": sample},
                "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
        print(json.dumps(line), flush=True)
        return

    import torch
    if world > 1:
        torch.distributed.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
    peak, peak_kind = measured_peaks()
    out_dir = Path(args.clocks_dir) if args.clocks_dir else Path(tempfile.gettempdir())
    out_dir.mkdir(parents=True, exist_ok=True)
    gpu_index = int(os.environ.get("LOCAL_RANK", "0"))
    sampler = ClockSampler(gpu_index, out_dir / f"clocks_rank{rank}.csv") if rank == 0 else None
    time.sleep(0.3 if sampler else 0)

    res = run_gpu(wl, args.steps, warmup, rank, args.e2e_steps if rank == 0 else 0,
                  flush_l2=algorithmic_bytes(wl) < 512e6)
    if world > 1:
        res["total_ms"] = max_over_ranks(res["total_ms"], "cuda")
        if res.get("l2_flushed"):  # timed per launch: the slowest rank's launch total
            res["launch_total_ms"] = max_over_ranks(sum(res["launch_ms"]), "cuda")
    clocks = sampler.summary(*res["wall"]) if sampler else None
    main_sum = summarize(wl, res, world, peak, peak_kind)

    secondary = []
    if args.secondary and rank == 0 and world == 1:
        for wl2 in parse_secondary(args.secondary):
            r2 = run_gpu(wl2, args.steps, warmup, rank, 0, flush_l2=algorithmic_bytes(wl2) < 512e6)
            s2 = summarize(wl2, r2, 1, peak, peak_kind)
            s2["clocks"] = sampler.summary(*r2["wall"]) if sampler else None
            secondary.append(s2)
    toy = run_toy(args.toy_steps) if (args.toy_steps and rank == 0 and world == 1) else None
    if sampler:
        sampler.stop()
    if rank != 0:
        if world > 1:
            torch.distributed.destroy_process_group()
        return

    got, dt, rate = time_oracle(wl, target_s=args.cpu_seconds)
    cpu = {"value": rate / 1e9, "unit": UNIT, "cores": 1, "nproc": os.cpu_count(), "kind": "oracle",
           "sample": f"one step over the first {got} elements of the {wl.name} list ({dt:.1f} s, single thread)"}
    cpu_lists = oracle_whole_lists(args.cpu_lists)

    details = out_dir / "bench_details.json"
    details.write_text(json.dumps({"main": main_sum, "secondary": secondary, "toy": toy, "clocks": clocks,
                                   "cpu_baseline": cpu, "cpu_lists": cpu_lists}, indent=1))
    line = result_line(wl, world, args.steps, warmup, l2_desc, main_sum, cpu, clocks, toy, details, secondary,
                       args.steps * res["launches_per_step"], cpu_lists)
    print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
