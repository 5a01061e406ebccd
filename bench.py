#!/usr/bin/env python3
"""Benchmark of the Blurry Window Attention prefill on GB300 through the C ABI.

One step = one bla_forward_chunked call (every kernel of the chunked forward) over the
long-context prefill workload: B=1, H=16, L=65536, d_k=d_v=128, M=128 modes, S=128 slots,
period T=4096, chunks of 128 tokens, bf16 inputs ~ N(0,1)/sqrt(d), seed = rank.  The metric is
prefill tokens/s (B*L tokens per step), summed over ranks (weak scaling: every rank runs its
own independent batch; there is no collective on the data path).

Printed (rank 0, one JSON line): the device-timed throughput with inputs resident in HBM,
the roofline of the dominant kernel (per-launch CUDA-event time on its launch stream, against
the measured bf16 peak), the end-to-end throughput through host buffers (H2D of q,k,v and D2H
of o inside the timed region), SM clocks sampled during timed work (the K steps and a sustained
leg of the same step looped for >= 1.5 s, reported beside them), the number of this
library's kernel launches in the timed region, the decode step's HBM roofline, and the float64
oracle timed on the host cores on a bounded sample of the same workload.

--impl reference times the float64 oracle alone (the method's reference implementation here)
on bounded samples of the same workload and prints the same line with "impl": "reference".
"""
import argparse
import math
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "BLA prefill tokens/s at 1 GB300 + %roofline (TC for prefill, HBM for decode)"
WORKLOAD = "prefill_bf16_long"
DECODE_WORKLOAD = "decode_bf16"


def canonical_flops(w, C=128):
    """Algorithmic contraction FLOPs per token-head of the chunked method, split by kernel.

    K pass: P = QK^T (2C dk), X = P E + Q W^T (2C R + 2 dk R), slot scores (2 R S), K state (2 R dk)
    V pass: U = p Phi (2 S R), G = A' E (2C R), O = G V + A' W_V (2C dv + 2 R dv), V state (2 R dv)
    with R = 2M-1 live state rows.  Their sum is 2C(dk+dv) + 4CR + 4RS + 4R(dk+dv).
    """
    R = 2 * w.M - 1
    dk = dv = w.d
    kpass = 2 * C * dk + 2 * C * R + 2 * dk * R + 2 * R * w.S + 2 * R * dk
    vpass = 2 * w.S * R + 2 * C * R + 2 * C * dv + 2 * R * dv + 2 * R * dv
    return {"kpass": kpass, "vpass": vpass, "total": kpass + vpass}


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


class ClockSampler:
    """nvidia-smi clock/throttle samples every 200 ms while running."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.rows = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu_id), "--query-gpu=" + self.FIELDS,
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        # nvidia-smi prints each sample as it takes it: the read time stamps the sample
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 8:
                self.rows.append((time.perf_counter(), parts))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        if self.thread is not None:
            self.thread.join(timeout=2)

    def summary(self, t0=None, t1=None):
        """Median SM clock, max clock and throttle reasons of the samples taken in [t0, t1]
        (perf_counter seconds; all samples when not given)."""
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for ts, r in self.rows:
            if (t0 is not None and ts < t0) or (t1 is not None and ts > t1):
                continue
            try:
                sm.append(float(r[0]))
                mx.append(float(r[1]))
            except ValueError:
                continue
            for name, val in zip(names, r[4:8]):
                if val.strip().lower() == "active":
                    reasons.add(name)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(n_gpus, backend="nccl"):
    """World size, rank and local rank from the torchrun environment; joins the process group
    (NCCL on GPUs; the CPU tests use gloo).  The group carries only timing reductions."""
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier_max(value, world):
    """The maximum of `value` over the ranks (the slowest rank's time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([value], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, units_per_rank, ms_max):
    """Weak scaling: every rank processes its own units; the job rate is all ranks' units over the
    slowest rank's time."""
    return world * units_per_rank / (ms_max / 1000.0)


def oracle_sample(w, budget_s, seed=0, form="naive"):
    """Time the float64 oracle on the first Ls tokens of every head of the workload, Ls sized
    so the run takes about budget_s seconds.  Returns (tokens/s, cores, sample description)."""
    import numpy as np
    import oracle
    from paper_2606_09862_gb300.inputs import make_qkv

    def run(Ls):
        q, k, v = make_qkv(w.B, w.H, Ls, w.d, dtype=w.dtype, seed=seed)
        t0 = time.perf_counter()
        oracle.forward(q, k, v, w.M, w.S, w.T, form=form)
        return time.perf_counter() - t0

    Ls = 16
    t = run(Ls)
    while t < budget_s / 4 and Ls < w.L:
        Ls = min(w.L, max(Ls * 2, int(Ls * budget_s / max(t, 1e-3) * 0.8)))
        t = run(Ls)
    cores = min(oracle.max_threads(), w.B * w.H)
    rate = w.B * Ls / t
    sample = ("float64 oracle (Alg. 2 recurrence, form=%s) on %d tokens x %d heads of the workload's shape "
              "and distribution (seeded), %.1f s" % (form, Ls, w.B * w.H, t))
    return rate, cores, sample, Ls, t


def run_reference(args):
    """--impl reference: the float64 oracle on bounded samples, rank 0 only."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    from paper_2606_09862_gb300.inputs import WORKLOADS
    import numpy as np
    import oracle
    from paper_2606_09862_gb300.inputs import make_qkv
    w = WORKLOADS[WORKLOAD]
    steps, warm = max(1, args.steps), max(0, args.warmup)
    per_step = max(0.2, args.ref_seconds / (steps + warm))
    # size one step's sample from a calibration run
    _, _, _, Ls, t = oracle_sample(w, per_step)
    q, k, v = make_qkv(w.B, w.H, Ls, w.d, dtype=w.dtype, seed=0)
    for _ in range(warm):
        oracle.forward(q, k, v, w.M, w.S, w.T, form="naive")
    times = []
    for _ in range(steps):
        t0 = time.perf_counter()
        oracle.forward(q, k, v, w.M, w.S, w.T, form="naive")
        times.append(time.perf_counter() - t0)
    ms = 1000.0 * statistics.mean(times)
    value = w.B * Ls / (ms / 1000.0)
    cores = min(oracle.max_threads(), w.B * w.H)
    sample = ("float64 oracle (Alg. 2 recurrence) over the first %d of %d tokens of all %d heads per step"
              % (Ls, w.L, w.B * w.H))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": steps, "warmup": warm, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD + ": B=1 H=16 L=65536 d=128 M=128 S=128 T=4096 chunk=128",
                       "sample_tokens_per_head": Ls},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def gpu_uuid(dev):
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(dev.index or 0)


def time_steps(fn, steps, stream):
    import torch
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    a.record(stream)
    for _ in range(steps):
        fn()
    b.record(stream)
    torch.cuda.synchronize()
    return a.elapsed_time(b) / steps


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="oracle CPU-baseline budget")
    ap.add_argument("--ref-seconds", type=float, default=120.0, help="total budget of --impl reference")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-decode", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--seq", type=int, default=0, help="override L (profiling captures of a smaller case)")
    ap.add_argument("--decode-batch", type=int, default=0, help="override the decode batch (profiling captures)")
    ap.add_argument("--no-configs", action="store_true", help="skip the timing of the other parity configs")
    ap.add_argument("--configs-only", default="",
                    help="comma-separated parity configs to time alone (profiling captures); prints their JSON")
    ap.add_argument("--configs-iters", type=int, default=20, help="timed calls per parity config")
    ap.add_argument("--no-sustained", action="store_true", help="skip the >= 1.5 s sustained leg (profiling captures)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.configs_only:
        return run_configs_only(args)

    import torch
    from paper_2606_09862_gb300 import bla
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_qkv, make_state, make_decode_step

    world, rank, local = dist_setup(args.gpus)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    w = WORKLOADS[WORKLOAD]
    if args.seq > 0:
        import dataclasses
        w = dataclasses.replace(w, L=args.seq)
    peaks = load_peaks()
    steps, warm = max(1, args.steps), max(3, args.warmup)

    # ---- inputs resident in HBM (805 MB of q, k, v > 129 MB L2: no flush needed)
    qh, kh, vh = (torch.from_numpy(x).to(torch.bfloat16) for x in make_qkv(w.B, w.H, w.L, w.d, "bf16", seed=rank))
    q, k, v = (x.to(dev) for x in (qh, kh, vh))
    o = torch.empty_like(v)
    lse = torch.empty((w.B, w.H, w.L), dtype=torch.float32, device=dev)
    p = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, dtype=torch.bfloat16)
    ws = torch.empty(bla.bla_workspace_bytes(p, bla.BLA_WS_FORWARD), dtype=torch.uint8, device=dev)

    def step():
        bla.bla_forward_chunked(q, k, v, w.M, w.S, w.T, workspace=ws, out=o, stream=stream)

    for _ in range(warm):
        step()
    bla.bla_device_error()

    # ---- timed region: device time with inputs resident
    sampler = ClockSampler(gpu_uuid(dev))
    sampler.start()
    time.sleep(0.3)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    n0 = bla.bla_kernel_launches()
    t_wall0 = time.perf_counter()
    ms = time_steps(step, steps, stream)
    wall = time.perf_counter() - t_wall0
    launches = bla.bla_kernel_launches() - n0
    if world > 1:
        torch.distributed.barrier()
    # ---- sustained leg: the same step back to back for >= 1.5 s, so that the clock samples (every
    # 200 ms) fall inside timed work and the power-capped clock is seen; reported beside the K steps
    sus_steps = 0 if args.no_sustained else max(steps, int(math.ceil(1500.0 / max(ms, 1e-3))))
    t_sus0 = time.perf_counter()
    sus_ms = time_steps(step, sus_steps, stream) if sus_steps else float("nan")
    t_sus1 = time.perf_counter()
    if world > 1:
        torch.distributed.barrier()
    sampler.stop()
    bla.bla_device_error()
    ms = barrier_max(ms, world)
    tokens_per_step = w.B * w.L
    value = whole_job_rate(world, tokens_per_step, ms)

    # ---- per-kernel launch times (same steps, CUDA events on the launch stream)
    bla.bla_profile_enable(True)
    prof_steps = min(steps, 20)
    for _ in range(prof_steps):
        step()
    torch.cuda.synchronize()
    prof = bla.bla_profile_collect()
    bla.bla_profile_enable(False)
    flops = canonical_flops(w)
    per_launch = {kname: ms_ / max(n, 1) for kname, (ms_, n) in prof.items()}
    dom = max(("kpass", "vpass"), key=lambda kname: per_launch.get(kname, 0.0))
    dom_ms = per_launch[dom]
    dom_flops = flops[dom] * w.B * w.H * w.L
    achieved = dom_flops / (dom_ms / 1000.0) / 1e12
    sustained = wall >= 1.0
    peak = peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"]
    traffic = stored_traffic(dom, w.L)
    roofline = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": traffic,
                "peak_kind": ("%s bf16 dense, %s" % ("sustained" if sustained else "burst", peaks["source"])),
                "flops_per_launch": dom_flops, "ms_per_launch": dom_ms,
                "kernels_ms_per_launch": per_launch,
                "step_frac_of_peak": flops["total"] * w.B * w.H * w.L / (ms / 1000.0) / 1e12 / peak}
    sus_ms = barrier_max(sus_ms, world) if sus_steps else None
    sustained_leg = None if not sus_steps else {"steps": sus_steps, "seconds": t_sus1 - t_sus0, "ms_per_step": sus_ms,
                     "value": whole_job_rate(world, tokens_per_step, sus_ms), "unit": "tokens/s",
                     "peak": peaks["bf16_tflops_sustained"],
                     "step_frac_of_sustained_peak": flops["total"] * w.B * w.H * w.L / (sus_ms / 1000.0) / 1e12 /
                     peaks["bf16_tflops_sustained"],
                     "clocks": sampler.summary(t_sus0, t_sus1)}

    # ---- end to end through host buffers (pinned), copies inside the timed region
    e2e = None
    if args.e2e_steps > 0:
        qp, kp, vp = (x.pin_memory() for x in (qh, kh, vh))
        oh = torch.empty(o.shape, dtype=o.dtype, pin_memory=True)
        bufs = {}
        bla.forward_from_host(qp, kp, vp, w.M, w.S, w.T, device=dev, bufs=bufs, out_host=oh)
        torch.cuda.synchronize()
        e_steps = args.e2e_steps
        t0 = time.perf_counter()
        for _ in range(e_steps):
            bla.forward_from_host(qp, kp, vp, w.M, w.S, w.T, device=dev, bufs=bufs, out_host=oh)
            torch.cuda.synchronize()      # the step's result is on the host
        e_ms = 1000.0 * (time.perf_counter() - t0) / e_steps
        e_ms = barrier_max(e_ms, world)
        e2e = {"value": whole_job_rate(world, tokens_per_step, e_ms), "unit": "tokens/s",
               "h2d_bytes_per_step": int(sum(x.numel() * x.element_size() for x in (qp, kp, vp))),
               "d2h_bytes_per_step": int(oh.numel() * oh.element_size()), "ms_per_step": e_ms}
        del bufs

    # ---- decode step: HBM roofline on the state bytes
    decode = None
    if not args.no_decode:
        dw = WORKLOADS[DECODE_WORKLOAD]
        if args.decode_batch > 0:
            import dataclasses
            dw = dataclasses.replace(dw, B=args.decode_batch)
        del q, k, v, o, ws
        torch.cuda.empty_cache()
        st = torch.from_numpy(make_state(dw.B, dw.H, dw.M, dw.d, dw.state_std, seed=rank)).to(dev)
        dq, dk, dv = (torch.from_numpy(x).to(torch.bfloat16).to(dev) for x in make_decode_step(0, dw.B, dw.H, dw.d,
                                                                                               "bf16", seed=rank))
        dpar = bla.make_params(dw.B, dw.H, 1, dw.d, dw.d, dw.M, dw.S, dw.T, dtype=torch.bfloat16)
        dws = torch.empty(bla.bla_workspace_bytes(dpar, bla.BLA_WS_DECODE), dtype=torch.uint8, device=dev)
        dout = torch.empty((dw.B, dw.H, dw.d), dtype=torch.bfloat16, device=dev)
        pos = [dw.decode_pos0]

        def dstep():
            bla.bla_decode_step(dq, dk, dv, st, pos[0], dw.M, dw.S, dw.T, workspace=dws, out=dout, stream=stream)
            pos[0] += 1

        for _ in range(3):
            dstep()
        bla.bla_profile_enable(True)
        d_ms = time_steps(dstep, 20, stream)
        dprof = bla.bla_profile_collect()
        bla.bla_profile_enable(False)
        bla.bla_device_error()
        k_ms = dprof["decode"][0] / max(dprof["decode"][1], 1)
        state_bytes = 2 * (2 * dw.d) * (2 * dw.M - 1) * 4 * dw.B * dw.H
        gbs = state_bytes / (k_ms / 1000.0) / 1e9
        decode = {"workload": DECODE_WORKLOAD + ": %d seqs x 16 heads, d=128, M=128, S=128, T=4096" % dw.B,
                  "tokens_per_s": dw.B / (d_ms / 1000.0), "ms_per_step": d_ms, "kernel_ms": k_ms,
                  "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                               "frac": gbs / peaks["hbm_gbs"], "bytes_per_launch": state_bytes}}

    # ---- the other parity configs (rank 0, N = 1 only)
    configs = None
    if rank == 0 and world == 1 and not args.no_configs and args.seq == 0:
        configs = measure_configs(bla, torch, dev, stream, peaks)

    # ---- CPU baseline: the oracle on a bounded sample (rank 0, N = 1 only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        rate, cores, sample, _, _ = oracle_sample(w, args.cpu_seconds)
        cpu = {"value": rate, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": steps,
                "warmup": warm, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": WORKLOAD + ": B=1 H=16 L=%d d_k=d_v=128 M=128 S=128 T=4096 chunk=128" % w.L,
                           "inputs": "q,k,v bf16 805 MB resident, larger than the 129 MB L2 (no flush)",
                           "accumulate": "fp32 (TMEM), state fp32"},
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
                "clocks": dict(sampler.summary(t_wall0, t_sus1), window="timed steps and the sustained leg"),
                "sustained": sustained_leg, "decode": decode, "configs": configs}
        print(json.dumps(line))
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_configs_only(args):
    """Time only the named parity configs (for ncu captures of their kernels) and print the JSON."""
    import torch
    from paper_2606_09862_gb300 import bla
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    names = tuple(n for n in args.configs_only.split(",") if n)
    out = measure_configs(bla, torch, dev, torch.cuda.current_stream(dev), load_peaks(), iters=max(1, args.configs_iters),
                          only=names, warm=max(1, min(3, args.warmup)))
    print(json.dumps({"configs": out}))
    return 0


def measure_configs(bla, torch, dev, stream, peaks, iters=20, only=None, warm=3):
    """The other parity configs, timed through the same ABI: config 2 (recall-shaped forward) and
    config 3 (LM-layer forward and backward).  Each call is timed alone with CUDA events after an
    L2 flush (config 2's inputs fit in L2); FLOPs are the canonical counts at chunk 64, the chunk
    the survey fixes for these configs' accounting; bytes are the tensors the call must read and
    write once."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_qkv, make_dout
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)   # 256 MB > 129 MB L2

    def timed(fn):
        for _ in range(warm):
            fn()
        tot = 0.0
        for _ in range(iters):
            flush.zero_()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            fn()
            b.record(stream)
            torch.cuda.synchronize()
            tot += a.elapsed_time(b)
        bla.bla_device_error()
        return tot / iters

    def roof(flops, nbytes, ms, tokens):
        tf = flops / (ms / 1000.0) / 1e12
        gbs = nbytes / (ms / 1000.0) / 1e9
        return {"ms": ms, "tokens_per_s": tokens / (ms / 1000.0), "tflops": tf, "gbs": gbs,
                "frac_tensor": tf / peaks["bf16_tflops"], "frac_hbm": gbs / peaks["hbm_gbs"],
                "bound": "hbm" if flops / nbytes < peaks["bf16_tflops"] * 1e3 / peaks["hbm_gbs"] else "tensor",
                "flops": flops, "bytes": nbytes}

    out = {}
    # the two parity configs in the lag form; config 3 and the long prefill also in the absolute
    # form (phase_mode "absolute", Alg. 1), which runs the same kernels with other tables
    for name, modes in (("fwd_bf16_recall", ("lag",)), ("fwdbwd_bf16_lm", ("lag", "absolute")),
                        ("prefill_bf16_long", ("absolute",))):
        if only:
            if name not in only:
                continue
            modes = ("lag",) if name != "prefill_bf16_long" else ("absolute",)
        w = WORKLOADS[name]
        q, k, v = (torch.from_numpy(x).to(torch.bfloat16).to(dev)
                   for x in make_qkv(w.B, w.H, w.L, w.d, "bf16", seed=0, recall_dup=getattr(w, "recall_dup", 0.0)))
        res = {}
        C = 64 if name != "prefill_bf16_long" else 128
        tok = w.B * w.L
        F = canonical_flops(w, C=C)["total"] * w.B * w.H * w.L
        elem = w.B * w.H * w.L * w.d
        for mode in modes:
            sfx = "" if mode == "lag" else "_absolute"
            par = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, dtype=torch.bfloat16, phase_mode=mode)
            ws = torch.empty(bla.bla_workspace_bytes(par, bla.BLA_WS_FORWARD), dtype=torch.uint8, device=dev)

            def fwd():
                return bla.bla_forward_chunked(q, k, v, w.M, w.S, w.T, workspace=ws, stream=stream, phase_mode=mode)

            res["forward" + sfx] = roof(F, 4 * elem * 2 + w.B * w.H * w.L * 4, timed(fwd), tok)
            if getattr(w, "backward", False):
                o, lse, _ = fwd()
                do = torch.from_numpy(make_dout(w.B, w.H, w.L, w.d, "bf16", seed=0)).to(torch.bfloat16).to(dev)
                bws = torch.empty(bla.bla_workspace_bytes(par, bla.BLA_WS_BACKWARD), dtype=torch.uint8, device=dev)

                def bwd():
                    return bla.bla_backward(q, k, v, o, do, lse, w.M, w.S, w.T, workspace=bws, stream=stream,
                                            phase_mode=mode)

                res["backward" + sfx] = roof(2 * F, 8 * elem * 2 + w.B * w.H * w.L * 4, timed(bwd), tok)
                del o, lse, do, bws
            del ws
        res["shape"] = "B=%d H=%d L=%d d=%d M=%d S=%d T=%d" % (w.B, w.H, w.L, w.d, w.M, w.S, w.T)
        out[name] = res
        del q, k, v
    if not only or "fwd_f32_small" in only:
        w = WORKLOADS["fwd_f32_small"]
        q, k, v = (torch.from_numpy(x).to(dev) for x in make_qkv(w.B, w.H, w.L, w.d, "f32", seed=0))
        par = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, chunk=w.chunk, dtype=torch.float32)
        wsf = torch.empty(bla.bla_workspace_bytes(par, bla.BLA_WS_FORWARD), dtype=torch.uint8, device=dev)
        ms = timed(lambda: bla.bla_forward_chunked(q, k, v, w.M, w.S, w.T, chunk=w.chunk, workspace=wsf))
        out["fwd_f32_small"] = {"forward": {"ms": ms, "tokens_per_s": w.B * w.L / (ms / 1000.0)},
                                "shape": "B=%d H=%d L=%d d=%d M=%d S=%d T=%g chunk=%d fp32" %
                                         (w.B, w.H, w.L, w.d, w.M, w.S, w.T, w.chunk)}
    if not only or "lm_block_f32" in only:
        out["lm_block_f32"] = measure_block(bla, torch, dev, timed)
    if not only or "decay_bf16_lm" in only:
        out["decay_bf16_lm"] = measure_decay(bla, torch, dev, timed, peaks)
    del flush
    torch.cuda.empty_cache()
    return out


def measure_block(bla, torch, dev, timed):
    """One BLA layer of the RegBench-sized LM block (d_model 128, 4 heads, M = 16, S = 31, T = 62,
    batch 32, L = 256; fp32): input projections (cuBLAS), token mixing (fp32 path), output projection."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_block_inputs
    from paper_2606_09862_gb300.layer import bla_block_forward
    w = WORKLOADS["lm_block_f32"]
    dm = w.H * w.d
    x, ws = make_block_inputs(w.B, w.L, dm, seed=0)
    x = torch.from_numpy(x).to(dev)
    ws = [torch.from_numpy(a).to(dev) for a in ws]
    par = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, dtype=torch.float32)
    wsp = torch.empty(bla.bla_workspace_bytes(par, bla.BLA_WS_FORWARD), dtype=torch.uint8, device=dev)
    mix = {}

    def layer():
        return bla_block_forward(x, *ws, w.H, w.M, w.S, w.T, workspace=wsp)

    def mixing():
        return bla.bla_forward_chunked(mix["q"], mix["k"], mix["v"], w.M, w.S, w.T, want_lse=False, workspace=wsp)

    mix["q"], mix["k"], mix["v"] = (torch.randn(w.B, w.H, w.L, w.d, device=dev) for _ in range(3))
    ms = timed(layer)
    ms_mix = timed(mixing)
    return {"layer_ms": ms, "mixing_ms": ms_mix, "tokens_per_s": w.B * w.L / (ms / 1000.0),
            "shape": "B=%d L=%d d_model=%d H=%d d=%d M=%d S=%d T=%g fp32" % (w.B, w.L, dm, w.H, w.d, w.M, w.S, w.T)}


# Nominal fp32 SIMT peak of the part: 152 SMs x 128 fp32 lanes x 2 flops (FMA) x 2.07 GHz.


def measure_decay(bla, torch, dev, timed, peaks):
    """The state decay of Sec. 3.3 (absolute form): the LM-layer prefill (B=8, H=8, L=4096, d=128,
    M=64, S=64, T=1024, bf16), its backward, and one decode step at B=256, H=16, d=128, M=128, S=128,
    T=4096, pos = 4096, from a random fp32 slot state.

    The forward and backward run the chunked kernels (warp-level bf16 MMAs for the contractions,
    triangle walks on the CUDA cores); they are bound by latency, not by a roof, so both fractions
    are reported.  FLOPs count the contractions per token and head (c = chunk length, S slots):
    forward (c = 64) P, Y, O and the two state updates, 4 c d + 8 S d; backward (c = 32) P, Y, PV,
    YV, dQ, the chunk parts of dK and dV, Z, the state pass and the adjoint pass,
    10 c d + 18 S d.  Bytes are the tensors a call must read and write once: q, k, v, o and lse
    forward; q, k, v, dO, lse, dq, dk, dv backward.  The decode reads and writes the whole slot
    state once."""
    from paper_2606_09862_gb300.inputs import WORKLOADS, make_decode_step, make_dout, make_qkv, make_slot_state
    w = WORKLOADS["decay_bf16_lm"]
    q, k, v = (torch.from_numpy(x).to(torch.bfloat16).to(dev) for x in make_qkv(w.B, w.H, w.L, w.d, "bf16", seed=0))
    par = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, dtype=torch.bfloat16, phase_mode="absolute")
    ws = torch.empty(bla.bla_workspace_bytes(par, bla.BLA_WS_DECAY_FORWARD), dtype=torch.uint8, device=dev)
    o = torch.empty_like(v)
    units = w.B * w.H * w.L

    def entry(ms, flops, nbytes):
        tf = flops / (ms / 1000.0) / 1e12
        gbs = nbytes / (ms / 1000.0) / 1e9
        return {"ms": ms, "tokens_per_s": w.B * w.L / (ms / 1000.0), "tflops": tf, "flops": flops, "gbs": gbs,
                "bytes": nbytes, "bound": "latency", "frac_tensor": tf / peaks["bf16_tflops"],
                "frac_hbm": gbs / peaks["hbm_gbs"]}

    ms = timed(lambda: bla.bla_decay_forward(q, k, v, w.M, w.S, w.T, workspace=ws, out=o))
    res = {"forward": entry(ms, float(units) * (4 * 64 * w.d + 8 * w.S * w.d), float(units) * (8 * w.d + 4)),
           "shape": "B=%d H=%d L=%d d=%d M=%d S=%d T=%d bf16 absolute+decay" % (w.B, w.H, w.L, w.d, w.M, w.S, w.T)}
    o, lse, _ = bla.bla_decay_forward(q, k, v, w.M, w.S, w.T, workspace=ws)
    do = torch.from_numpy(make_dout(w.B, w.H, w.L, w.d, "bf16", seed=0)).to(torch.bfloat16).to(dev)
    parb = bla.make_params(w.B, w.H, w.L, w.d, w.d, w.M, w.S, w.T, dtype=torch.bfloat16, phase_mode="absolute")
    wsb = torch.empty(bla.bla_workspace_bytes(parb, bla.BLA_WS_DECAY_BACKWARD), dtype=torch.uint8, device=dev)
    ms_b = timed(lambda: bla.bla_decay_backward(q, k, v, o, do, lse, w.M, w.S, w.T, workspace=wsb))
    res["backward"] = entry(ms_b, float(units) * (10 * 32 * w.d + 18 * w.S * w.d), float(units) * (14 * w.d + 4))
    del q, k, v, ws, o, lse, do, wsb
    wd = WORKLOADS["decay_decode_bf16"]
    qd, kd, vd = (torch.from_numpy(x).to(torch.bfloat16).to(dev)
                  for x in make_decode_step(0, wd.B, wd.H, wd.d, "bf16", seed=0))
    st = torch.from_numpy(make_slot_state(wd.B, wd.H, wd.S, wd.d, wd.state_std, seed=0)).to(dev)
    pard = bla.make_params(wd.B, wd.H, 1, wd.d, wd.d, wd.M, wd.S, wd.T, dtype=torch.bfloat16, phase_mode="absolute")
    wsd = torch.empty(max(bla.bla_workspace_bytes(pard, bla.BLA_WS_DECAY_DECODE), 1), dtype=torch.uint8, device=dev)
    od = torch.empty((wd.B, wd.H, wd.d), dtype=torch.bfloat16, device=dev)
    ms_d = timed(lambda: bla.bla_decay_decode_step(qd, kd, vd, st, wd.decode_pos0, wd.M, wd.S, wd.T, workspace=wsd,
                                                   out=od))
    nbytes = 2 * st.numel() * 4 + 4 * wd.B * wd.H * wd.d * 2
    gbs = nbytes / (ms_d / 1000.0) / 1e9
    res["decode"] = {"ms": ms_d, "tokens_per_s": wd.B / (ms_d / 1000.0), "gbs": gbs, "bytes": nbytes,
                     "bound": "hbm", "frac_hbm": gbs / peaks["hbm_gbs"],
                     "shape": "B=%d H=%d d=%d M=%d S=%d T=%d pos=%d bf16, fp32 slot state" %
                              (wd.B, wd.H, wd.d, wd.M, wd.S, wd.T, wd.decode_pos0)}
    del qd, kd, vd, st, wsd, od
    return res


def stored_traffic(kernel, L):
    """DRAM bytes per launch (read + write) of `kernel` from profiles/traffic_<kernel>.txt, written
    from an ncu capture, scaled to L tokens; None if absent or if the CUDA sources changed since."""
    path = os.path.join(ROOT, "profiles", "traffic_%s.txt" % kernel)
    if not os.path.exists(path):
        return None
    kv = {}
    with open(path) as f:
        for line in f:
            if "=" in line and not line.startswith("#"):
                a, b = line.split("=", 1)
                kv[a.strip()] = b.strip()
    if kv.get("source_digest") != _source_digest():
        return None
    try:
        return float(kv["bytes_per_launch"]) * L / float(kv["tokens_per_head"])
    except (KeyError, ValueError):
        return None


# The sources the chunked passes (K and V pass) are compiled from.
PASS_SOURCES = ("common.cuh", "fwd_bf16.cu", "fwd_bf16.cuh", "tc.cuh", "tmap.cu", "tmap.cuh")


def _strip_comments(src):
    """C/C++ source without its // and /* */ comments (string and character literals kept)."""
    out, i, n = [], 0, len(src)
    while i < n:
        c = src[i]
        if c in "\"'":
            j = i + 1
            while j < n and src[j] != c:
                j += 2 if src[j] == "\\" else 1
            out.append(src[i:j + 1])
            i = j + 1
        elif src.startswith("//", i):
            j = src.find("\n", i)
            i = n if j < 0 else j
        elif src.startswith("/*", i):
            j = src.find("*/", i + 2)
            i = n if j < 0 else j + 2
        else:
            out.append(c)
            i += 1
    return "".join(out)


def _source_digest():
    """Digest of the sources of the chunked passes with comments removed and whitespace runs
    collapsed; a stored DRAM-traffic figure of a pass is used only if it matches (any change to the
    code of those files may change the pass kernels, a change to a comment or a line break does
    not)."""
    import hashlib
    h = hashlib.sha256()
    d = os.path.join(ROOT, "paper_2606_09862_gb300", "csrc")
    for fn in PASS_SOURCES:
        with open(os.path.join(d, fn), encoding="utf-8") as f:
            h.update(fn.encode())
            h.update(" ".join(_strip_comments(f.read()).split()).encode())
    return h.hexdigest()[:16]


if __name__ == "__main__":
    sys.exit(main())
