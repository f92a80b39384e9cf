"""Benchmark: fwd+bwd tokens/s of sliced causal Performer attention on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--C C] [--sweep]

A step is one slim_fwd + slim_bwd over the whole workload (every chain, every
slice).  The default workload is B=8 H=8 L=4096 d=64 M=256, bf16 inputs, fp32
accumulation, FAVOR+ features, slice C=1024.  Rank 0 prints ONE JSON line.

Under torchrun (N > 1) every rank runs an independent replica of the workload
on its own GPU (the chains are independent; there is no data-path
collective), timing is bracketed by barriers and the max over ranks is used.

--impl reference times the fp64 CPU oracle (the slow, obviously-correct
program the CUDA path is checked against) on the host cores, on the same
workload and metric, each step a bounded sample of chains.

--sweep prints one JSON line per slice size of the L=32768 workload
(tokens/s and peak device memory vs C); it is not the default line.
"""
import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "fwd+bwd tokens/s at L=4096 H=8 d=64 M=256; % roofline; peak mem vs slice C"
DEFAULT_WORKLOAD = "L4096_bf16"
L2_BYTES = 129 * 1024 * 1024
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# FP32 FMA issue rate: 152 SMs x 128 lanes x 2 FLOP x 2.07 GHz (maximum SM clock)
FP32_ALU_TFLOPS = 152 * 128 * 2 * 2.07e9 / 1e12
# MUFU exponentials: ex2.approx.f32 measured on this machine's GB300 with 8
# independent chains per thread over 1216 CTAs of 256 threads: 9.5e12 per
# second, 30 per clock per SM at 2070 MHz
MUFU_EX2_PER_S = 9.5e12

# roofline bound of each kernel: (bound, which algorithmic quantity)
KERNEL_BOUND = {
    "simt_gemm": ("alu", "flops"),
    "simt_prep": ("alu", "flops"),
    "tc_fwd": ("tensor", "flops"),
    "tc_bwd": ("tensor", "flops"),
    "tc_bwd_q": ("tensor", "flops"),
    "tc_bwd_kv": ("tensor", "flops"),
    "tc_delta": ("tensor", "flops"),
}


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--C", type=int, default=None)
    # shape overrides, for profiling a smaller case of a workload (ncu captures)
    ap.add_argument("--B", type=int, default=None)
    ap.add_argument("--H", type=int, default=None)
    ap.add_argument("--sweep", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    return ap.parse_args()


# ------------------------------------------------------------------ distributed
def dist_setup():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    if ws <= 1:
        return 0, 1, 0
    import torch
    import torch.distributed as dist
    rank = int(os.environ["RANK"])
    local = int(os.environ.get("LOCAL_RANK", rank))
    backend = "nccl" if torch.cuda.is_available() else "gloo"
    if backend == "nccl":
        torch.cuda.set_device(local)
    dist.init_process_group(backend=backend)
    return rank, ws, local


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, ws):
    """Largest value of x over all ranks (timing only; no data-path use)."""
    if ws <= 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x, ws):
    if ws <= 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([float(x)], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi sampled every 50 ms while the timed region runs."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.lines = []
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu_id), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.12)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, smax, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for n, p in zip(names, parts[5:9]):
                if p.lower().startswith("active"):
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "samples": len(sm), "reasons": sorted(reasons)}


def gpu_id_for(dev_index):
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev_index).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return dev_index


# ------------------------------------------------------------------ peaks / roofline
def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return FALLBACK_PEAKS, "fallback"


def traffic_for(kernel):
    """DRAM bytes per launch from the committed ncu summary, if the kernel's
    source is unchanged since the capture (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        table = json.load(f)
    ent = table.get(kernel)
    if not ent:
        return None
    import hashlib
    src = os.path.join(ROOT, ent["source"])
    if not os.path.exists(src):
        return None
    with open(src, "rb") as f:
        if hashlib.sha256(f.read()).hexdigest() != ent["source_sha256"]:
            return None
    return ent["dram_bytes_per_launch"]


def roofline(stats, steps):
    peaks, which = measured_peaks()
    top = max(stats, key=lambda s: s["total_ms"]) if stats else None
    if top is None or top["launches"] == 0:
        return None
    bound, qty = KERNEL_BOUND.get(top["name"], ("hbm", "bytes"))
    avg_s = top["total_ms"] / top["launches"] / 1e3
    per_launch = top[qty] / top["launches"]
    if bound == "hbm":
        achieved, peak, unit = per_launch / avg_s / 1e9, peaks["hbm_gbs"], "GB/s"
        peak_note = f"{which} hbm_gbs"
    elif bound == "tensor":
        achieved, peak, unit = per_launch / avg_s / 1e12, peaks["bf16_tflops"], "TFLOP/s"
        peak_note = f"{which} bf16_tflops (burst)"
    else:
        achieved, peak, unit = per_launch / avg_s / 1e12, FP32_ALU_TFLOPS, "TFLOP/s"
        peak_note = "fp32 FMA issue rate at 2.07 GHz (derived)"
    total_ms = sum(s["total_ms"] for s in stats)
    return {"bound": bound, "achieved": round(achieved, 3), "peak": round(peak, 1), "unit": unit,
            "frac": round(achieved / peak, 4), "traffic": traffic_for(top["name"]),
            "kernel": top["name"], "peak_source": peak_note,
            "launches_per_step": top["launches"] / steps,
            "avg_launch_us": round(avg_s * 1e6, 3),
            "share_of_kernel_time": round(top["total_ms"] / total_ms, 4) if total_ms else None}


def step_ceilings(w, B, H, L, ms_per_step):
    """The three floors of one fwd+bwd step from its algorithmic work per
    token-head: 30dM FLOPs (on the tensor pipe for bf16, the FP32 FMA pipe
    otherwise), 12ds HBM bytes (s = element size) and 4M exponentials (exp
    features; none for ReLU), against the measured peaks."""
    peaks, which = measured_peaks()
    th = B * H * L
    flops = 30.0 * w.d * w.M * th
    s = 2 if w.dtype == "bf16" else 4
    hbm_bytes = 12.0 * w.d * s * th
    exps = 4.0 * w.M * th if w.feature == "exp" else 0.0
    if w.dtype == "bf16":
        compute_us, compute = flops / (peaks["bf16_tflops"] * 1e12) * 1e6, "tensor"
    else:
        compute_us, compute = flops / (FP32_ALU_TFLOPS * 1e12) * 1e6, "fp32 alu"
    floors = {compute: compute_us, "hbm": hbm_bytes / (peaks["hbm_gbs"] * 1e9) * 1e6,
              "mufu": exps / MUFU_EX2_PER_S * 1e6}
    bound = max(floors, key=floors.get)
    return {"floors_us": {k: round(v, 2) for k, v in floors.items()}, "bound": bound,
            "t_star_us": round(floors[bound], 2),
            "frac_of_step": round(floors[bound] / (ms_per_step * 1e3), 4),
            "flops": flops, "hbm_bytes": hbm_bytes, "exps": exps,
            "peak_source": f"{which} peaks; mufu {MUFU_EX2_PER_S:.2e}/s measured"}


# ------------------------------------------------------------------ CPU oracle
def _oracle_chain(args):
    """One chain's fp64 oracle fwd+bwd (runs in a spawned worker)."""
    name, overrides, b, h = args
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    import oracle
    from paper_2012_11346_gb300 import workloads as W
    w = W.WORKLOADS[name].with_(**overrides)
    x = W.make_inputs(w)
    c = {n: W.as_float64_numpy(t[b:b + 1, h:h + 1] if t.dim() == 4 else t) for n, t in x.items()}
    t0 = time.perf_counter()
    o, S, z = oracle.oracle_fwd(c["q"], c["k"], c["v"], c["omega"], w.C, w.feature)
    oracle.oracle_bwd(c["q"], c["k"], c["v"], c["omega"], c["dout"], S, z, w.C, w.feature)
    return time.perf_counter() - t0


def oracle_pool_size():
    return max(1, min(len(os.sched_getaffinity(0)), 16))


def _pool_warm(_):
    """Imports what the oracle workers need, then holds the worker briefly so
    that the other workers take the remaining items."""
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    import oracle  # noqa: F401
    from paper_2012_11346_gb300 import workloads  # noqa: F401
    time.sleep(0.2)
    return os.getpid()


def start_oracle_pool(n):
    """A spawned pool whose workers have finished starting up and importing,
    so that no worker start-up competes with the GPU timing for host cores."""
    import multiprocessing as mp
    pool = mp.get_context("spawn").Pool(n)
    pool.map(_pool_warm, range(n), chunksize=1)
    return pool


def oracle_sample(w, overrides, pool, nchains):
    """Runs nchains chains of the workload through the oracle in parallel;
    returns (tokens, wall seconds)."""
    jobs = [(w.name, overrides, (i // w.H) % w.B, i % w.H) for i in range(nchains)]
    secs = pool.map(_oracle_chain, jobs)
    # the chains run side by side; input generation is outside each worker's clock
    return nchains * w.L, max(secs)


# ------------------------------------------------------------------ our arm
def run_ours(args, rank, ws, local):
    import torch
    from paper_2012_11346_gb300 import slim
    from paper_2012_11346_gb300 import workloads as W


    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = W.WORKLOADS[args.workload]
    if args.C:
        w = w.with_(C=args.C)
    if args.B:
        w = w.with_(B=args.B)
    if args.H:
        w = w.with_(H=args.H)
    x = W.make_inputs(w, device=dev)
    q, k, v, om, dout = x["q"], x["k"], x["v"], x["omega"], x["dout"]
    B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
    out = torch.empty_like(q)
    S = torch.empty(B, H, M, d, dtype=torch.float32, device=dev)
    z = torch.empty(B, H, M, dtype=torch.float32, device=dev)
    S_lo, z_lo = torch.empty_like(S), torch.empty_like(z)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    dom = torch.empty(M, d, dtype=torch.float32, device=dev)
    wsf = torch.empty(max(256, slim.workspace_size(B, H, L, d, M, w.C, q.dtype, w.feature, False)),
                      dtype=torch.uint8, device=dev)
    wsb = torch.empty(max(256, slim.workspace_size(B, H, L, d, M, w.C, q.dtype, w.feature, True)),
                      dtype=torch.uint8, device=dev)

    def step():
        slim.forward_into(q, k, v, om, w.C, w.feature, out, S, z, wsf, S_lo=S_lo, z_lo=z_lo)
        slim.backward_into(q, k, v, om, out, dout, S, z, w.C, w.feature, dq, dk, dv, dom, wsb,
                           S_lo=S_lo, z_lo=z_lo)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    # headline: K steps, nothing recorded between the kernels
    sampler = ClockSampler(gpu_id_for(local))
    sampler.start()
    time.sleep(0.1)
    launches0 = slim.launch_count()
    barrier(ws)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(ws)
    launches = slim.launch_count() - launches0
    clocks = sampler.stop()
    slim.check_device_error(wsf)
    slim.check_device_error(wsb)
    ms = max_over_ranks(e0.elapsed_time(e1), ws)
    tokens = sum_over_ranks(B * L * args.steps, ws)
    value = tokens / (ms / 1e3)

    # per-kernel CUDA events: the same K steps again with every launch bracketed
    slim.profiler_reset()
    slim.profiler_enable(True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    slim.profiler_enable(False)
    ms_profiled = e0.elapsed_time(e1)
    stats = slim.profiler_read()
    # a bounded device wait that gave up would make the timings meaningless
    slim.check_device_error(wsf)
    slim.check_device_error(wsb)

    # untimed validation pass: every call clears the device error word at its
    # start, so check it after each step; a bounded wait that gave up during
    # the measurement would make the numbers above meaningless
    for _ in range(args.steps):
        step()
        slim.check_device_error(wsf)
        slim.check_device_error(wsb)

    # end to end through the public API: pinned host inputs in, results out
    hq, hk, hv, hdo = (t.cpu().pin_memory() for t in (q, k, v, dout))
    hom = om.cpu().pin_memory()
    hout, hdq, hdk, hdv = (torch.empty(q.shape, dtype=q.dtype).pin_memory() for _ in range(4))
    hdom = torch.empty(M, d, dtype=torch.float32).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in (hq, hk, hv, hdo, hom))
    d2h = sum(t.numel() * t.element_size() for t in (hout, hdq, hdk, hdv, hdom))

    def e2e_step():
        for dst, src in ((q, hq), (k, hk), (v, hv), (dout, hdo), (om, hom)):
            dst.copy_(src, non_blocking=True)
        step()
        for dst, src in ((hout, out), (hdq, dq), (hdk, dk), (hdv, dv), (hdom, dom)):
            dst.copy_(src, non_blocking=True)

    for _ in range(args.warmup):
        e2e_step()
    barrier(ws)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(args.steps):
        e2e_step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(ws)
    ms_e2e = max_over_ranks(e0.elapsed_time(e1), ws)
    e2e_value = tokens / (ms_e2e / 1e3)

    # peak device memory of one fwd+bwd through the allocating API
    del hq, hk, hv, hdo
    torch.cuda.synchronize()
    torch.cuda.reset_peak_memory_stats(dev)
    base = torch.cuda.memory_allocated(dev)
    o2, S2, z2, S2l, z2l = slim.forward(q, k, v, om, w.C, w.feature, residuals=True)
    g2 = slim.backward(q, k, v, om, o2, dout, S2, z2, w.C, w.feature, S_lo=S2l, z_lo=z2l)
    torch.cuda.synchronize()
    peak = torch.cuda.max_memory_allocated(dev)
    del o2, S2, z2, S2l, z2l, g2

    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": path_dtype(stats, w), "data": "synthetic",
        "config": {"workload": w.name, "B": B, "H": H, "L": L, "d": d, "M": M, "C": w.C,
                   "feature": w.feature, "input_dtype": w.dtype,
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                   "l2": "no flush; per-step working set (q,k,v,dout,out,dq,dk,dv) "
                         f"{8 * q.numel() * q.element_size() / 2**20:.0f} MiB > L2 129 MiB"},
        "e2e": {"value": round(e2e_value, 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": int(launches),
        "roofline": roofline(stats, args.steps),
        "ceilings": step_ceilings(w, B, H, L, ms / args.steps),
        "profiled_ms_per_step": round(ms_profiled / args.steps, 4),
        "clocks": clocks,
        "peak_mem": {"bytes": peak, "above_inputs_bytes": peak - base,
                     "workspace_bytes": wsb.numel()},
        "kernels": [{k_: (round(v_, 4) if isinstance(v_, float) else v_) for k_, v_ in s.items()}
                    for s in stats],
    }
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        # The oracle pool starts only after every GPU measurement: with an
        # idle pool alive during the GPU passes, the end-to-end pass was
        # measured ~400x slower on a 16-core host.  Spawned workers do not
        # inherit the parent's CUDA context.
        n = oracle_pool_size()
        pool = start_oracle_pool(n)
        tok, sec = oracle_sample(w, {"C": w.C}, pool, n)
        line["cpu_baseline"] = {"value": round(tok / sec, 2), "unit": "tokens/s", "cores": n,
                                "kind": "oracle",
                                "sample": f"{n} chains x L={L} of this workload, fp64 NumPy, "
                                          f"one spawned process per chain, {sec:.1f} s wall"}
        pool.close()
    if rank == 0:
        print(json.dumps(line), flush=True)


def path_dtype(stats, w):
    names = {s["name"] for s in stats}
    if any(n.startswith("tc_") for n in names):
        return "bf16"
    return "f32"


# ------------------------------------------------------------------ reference arm
def run_reference(args, rank, ws):
    if rank != 0:
        return
    import multiprocessing as mp
    from paper_2012_11346_gb300 import workloads as W
    w = W.WORKLOADS[args.workload]
    if args.C:
        w = w.with_(C=args.C)
    if args.B:
        w = w.with_(B=args.B)
    if args.H:
        w = w.with_(H=args.H)
    n = oracle_pool_size()
    with mp.get_context("spawn").Pool(n) as pool:
        for _ in range(args.warmup):
            oracle_sample(w, {"C": w.C}, pool, n)
        tok, sec = 0, 0.0
        for _ in range(args.steps):
            t, s = oracle_sample(w, {"C": w.C}, pool, n)
            tok += t
            sec += s
    value = tok / sec
    sample = (f"each step: {n} chains x L={w.L} of the workload through the fp64 NumPy oracle, "
              f"one spawned process per chain")
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 2), "unit": "tokens/s",
        "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(1e3 * sec / args.steps, 2), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "H": w.H, "L": w.L, "d": w.d, "M": w.M,
                   "C": w.C, "feature": w.feature, "input_dtype": w.dtype},
        "cpu_baseline": {"value": round(value, 2), "unit": "tokens/s", "cores": n,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": round(value, 2), "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ C sweep
def run_sweep(args, local):
    import torch
    from paper_2012_11346_gb300 import slim
    from paper_2012_11346_gb300 import workloads as W
    dev = torch.device("cuda", local)
    w0 = W.WORKLOADS["L32768_bf16"]
    x = W.make_inputs(w0, device=dev)
    floor = sum(t.numel() * t.element_size() for t in x.values()) + \
        4 * x["q"].numel() * x["q"].element_size()   # + out, dq, dk, dv
    for C in W.C_SWEEP:
        w = w0.with_(C=C)

        def step():
            o, S, z, Sl, zl = slim.forward(x["q"], x["k"], x["v"], x["omega"], C, w.feature,
                                           residuals=True)
            slim.backward(x["q"], x["k"], x["v"], x["omega"], o, x["dout"], S, z, C, w.feature,
                          S_lo=Sl, z_lo=zl)

        for _ in range(max(1, args.warmup)):
            step()
        torch.cuda.synchronize()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(args.steps):
            step()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / args.steps
        peak = torch.cuda.max_memory_allocated(dev)
        # lower-bound point (Sec. 4.1): the same method on an input of length C only
        xl = {n: (t[:, :, :C].contiguous() if t.dim() == 4 else t) for n, t in x.items()}
        torch.cuda.synchronize()
        torch.cuda.reset_peak_memory_stats(dev)
        base_lb = torch.cuda.memory_allocated(dev)
        o, S, z, Sl, zl = slim.forward(xl["q"], xl["k"], xl["v"], xl["omega"], C, w.feature,
                                       residuals=True)
        slim.backward(xl["q"], xl["k"], xl["v"], xl["omega"], o, xl["dout"], S, z, C, w.feature,
                      S_lo=Sl, z_lo=zl)
        torch.cuda.synchronize()
        lb_above = torch.cuda.max_memory_allocated(dev) - base_lb
        del xl, o, S, z, Sl, zl
        print(json.dumps({"sweep": "L32768_bf16", "C": C, "tokens_per_s": round(w.B * w.L / (ms / 1e3), 1),
                          "ms_per_step": round(ms, 3), "peak_mem_bytes": peak,
                          "peak_above_inputs_bytes": peak - base, "io_floor_bytes": floor,
                          "length_C_input_above_inputs_bytes": lb_above,
                          "fwd_ws_bytes": slim.workspace_size(w.B, w.H, w.L, w.d, w.M, C,
                                                              x["q"].dtype, w.feature, False),
                          "bwd_ws_bytes": slim.workspace_size(w.B, w.H, w.L, w.d, w.M, C,
                                                              x["q"].dtype, w.feature, True)}),
              flush=True)


def main():
    args = parse()
    rank, ws, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, rank, ws)
    elif args.sweep:
        if rank == 0:
            run_sweep(args, local)
    else:
        run_ours(args, rank, ws, local)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
