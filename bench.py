"""Benchmark: fwd+bwd tokens/s of sliced causal Performer attention on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--C C] [--mode causal|bidir|segments]
                    [--segments S] [--sweep]

A step is one slim_fwd + slim_bwd over the whole workload (every chain, every
slice).  The default workload is B=8 H=8 L=4096 d=64 M=256, bf16 inputs, fp32
accumulation, FAVOR+ features, slice C=1024.  Rank 0 prints ONE JSON line; on
the default workload it carries `mem_vs_C`, the time and peak memory of the
B2 H8 L32768 workload for each slice size C.  --mode bidir times the
non-causal form instead, --mode segments the causal sweeps over S chained
segment calls (slim_fwd_from / slim_bwd_from).

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
    "mma_gemm": ("tensor", "flops"),
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
    ap.add_argument("--no-mem-curve", action="store_true")
    # what one step runs: the causal sweeps (default), the non-causal form, or
    # the causal sweeps over --segments chained calls (streaming)
    ap.add_argument("--mode", choices=["causal", "bidir", "segments", "stack"], default="causal")
    ap.add_argument("--segments", type=int, default=4)
    ap.add_argument("--layers", type=int, default=3)
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
    token-head: 30dM FLOPs (on the tensor pipe for bf16; for fp32 as six
    products of bf16 pieces on the tensor pipe), 12ds HBM bytes (s = element size) and 4M exponentials (exp
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
        # fp32 products on the tensor pipe as 6 products of bf16 pieces (24-bit
        # operands), the faster of that and the FP32 FMA pipe
        compute_us, compute = min(
            (flops * 6 / (peaks["bf16_tflops"] * 1e12) * 1e6, "tensor x6"),
            (flops / (FP32_ALU_TFLOPS * 1e12) * 1e6, "fp32 alu"))
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
    """One chain's fp64 oracle fwd+bwd (runs in a spawned worker); the
    non-causal form for mode bidir, the causal sweeps otherwise."""
    name, overrides, b, h, mode, layers = args
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    import oracle
    from paper_2012_11346_gb300 import workloads as W
    w = W.WORKLOADS[name].with_(**overrides)
    x = W.make_inputs(w)
    c = {n: W.as_float64_numpy(t[b:b + 1, h:h + 1] if t.dim() == 4 else t) for n, t in x.items()}
    if mode == "stack":
        xs = W.make_stack_inputs(w, layers)
        sx = W.as_float64_numpy(xs["x"][b:b + 1, h:h + 1])
        sdy = W.as_float64_numpy(xs["dy"][b:b + 1, h:h + 1])
        oms = list(W.as_float64_numpy(xs["omegas"]))
        t0 = time.perf_counter()
        y, S, z = oracle.oracle_stack_fwd(sx, oms, w.C, w.feature)
        oracle.oracle_stack_bwd(sx, oms, sdy, S, z, w.C, w.feature)
        return time.perf_counter() - t0
    t0 = time.perf_counter()
    if mode == "bidir":
        o, S, z = oracle.oracle_bidir_fwd(c["q"], c["k"], c["v"], c["omega"], w.C, w.feature)
        oracle.oracle_bidir_bwd(c["q"], c["k"], c["v"], c["omega"], c["dout"], S, z, w.C,
                                w.feature)
    else:
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


def oracle_sample(w, overrides, pool, nchains, mode="causal", layers=3):
    """Runs nchains chains of the workload through the oracle in parallel;
    returns (tokens, wall seconds)."""
    jobs = [(w.name, overrides, (i // w.H) % w.B, i % w.H, mode, layers) for i in range(nchains)]
    secs = pool.map(_oracle_chain, jobs)
    # the chains run side by side; input generation is outside each worker's clock
    return nchains * w.L, max(secs)


# ------------------------------------------------------------------ our arm
class StepSet:
    """Device buffers of one step and the calls that make it.  mode causal:
    slim_fwd + slim_bwd (with the forward's residuals); bidir: the non-causal
    pair; segments: the sequence cut into `segments` contiguous segments, the
    forwards chained through slim_fwd_from and the backwards, last segment
    first, through slim_bwd_from (each hands G^(0) to the one before)."""

    def __init__(self, w, dev, mode, segments, x=None, layers=3):
        import torch
        from paper_2012_11346_gb300 import slim
        from paper_2012_11346_gb300 import workloads as W
        self.w, self.mode, self.slim = w, mode, slim
        self.x = x if x is not None else W.make_inputs(w, device=dev)
        B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
        q = self.x["q"]
        f32 = torch.float32
        self.om = None if w.feature == "square" else self.x["omega"]
        if mode == "stack":
            # s residual layers by Algorithm 1: x, per-layer Omegas, dy
            self.layers = layers
            self.sx = W.make_stack_inputs(w, layers, device=dev)
            self.soms = None if w.feature == "square" else self.sx["omegas"]
            B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
            self.y = torch.empty_like(self.sx["x"])
            self.dx = torch.empty_like(self.sx["x"])
            self.sS = torch.empty(layers, B, H, M, d, dtype=f32, device=dev)
            self.sz = torch.empty(layers, B, H, M, dtype=f32, device=dev)
            self.sSl, self.szl = torch.empty_like(self.sS), torch.empty_like(self.sz)
            self.sdom = torch.empty(layers, M, d, dtype=f32, device=dev)
            size = slim.stack_workspace_size
            self.ws_f = self._ws(size(B, H, L, d, M, w.C, layers, q.dtype, w.feature, False), dev)
            self.ws_b = self._ws(size(B, H, L, d, M, w.C, layers, q.dtype, w.feature, True), dev)
            self.outputs = [self.y, self.dx, self.sdom]
            self.inputs = [self.sx["x"], self.sx["dy"], self.sx["omegas"]]
            return
        if mode == "segments":
            cuts = [round(i * L / segments) for i in range(segments + 1)]
            self.segs = []
            for a, b in zip(cuts[:-1], cuts[1:]):
                sg = {n: self.x[n][:, :, a:b].contiguous() for n in ("q", "k", "v", "dout")}
                sg.update(out=torch.empty_like(sg["q"]), dq=torch.empty_like(sg["q"]),
                          dk=torch.empty_like(sg["q"]), dv=torch.empty_like(sg["q"]),
                          S=torch.empty(B, H, M, d, dtype=f32, device=dev),
                          z=torch.empty(B, H, M, dtype=f32, device=dev),
                          S_lo=torch.empty(B, H, M, d, dtype=f32, device=dev),
                          z_lo=torch.empty(B, H, M, dtype=f32, device=dev),
                          G=torch.empty(B, H, M, d, dtype=f32, device=dev),
                          gz=torch.empty(B, H, M, dtype=f32, device=dev),
                          dom=torch.empty(M, d, dtype=f32, device=dev))
                self.segs.append(sg)
            Lmax = max(b - a for a, b in zip(cuts[:-1], cuts[1:]))
            self.ws_f = self._ws(slim.workspace_size(B, H, Lmax, d, M, w.C, q.dtype, w.feature,
                                                     False), dev)
            self.ws_b = self._ws(slim.workspace_size(B, H, Lmax, d, M, w.C, q.dtype, w.feature,
                                                     True), dev)
            self.outputs = [t for sg in self.segs for t in (sg["out"], sg["dq"], sg["dk"],
                                                            sg["dv"], sg["dom"])]
            self.inputs = [t for sg in self.segs for t in (sg["q"], sg["k"], sg["v"],
                                                           sg["dout"])] + [self.x["omega"]]
            return
        self.out = torch.empty_like(q)
        self.S = torch.empty(B, H, M, d, dtype=f32, device=dev)
        self.z = torch.empty(B, H, M, dtype=f32, device=dev)
        self.S_lo, self.z_lo = torch.empty_like(self.S), torch.empty_like(self.z)
        self.dq, self.dk, self.dv = (torch.empty_like(q) for _ in range(3))
        self.dom = torch.empty(M, d, dtype=f32, device=dev)
        if mode == "bidir":
            size = slim.bidir_workspace_size
            self.ws_f = self._ws(size(B, H, L, d, M, w.C, q.dtype, w.feature, False), dev)
            self.ws_b = self._ws(size(B, H, L, d, M, w.C, q.dtype, w.feature, True), dev)
        else:
            size = slim.workspace_size
            self.ws_f = self._ws(size(B, H, L, d, M, w.C, q.dtype, w.feature, False), dev)
            self.ws_b = self._ws(size(B, H, L, d, M, w.C, q.dtype, w.feature, True), dev)
        self.outputs = [self.out, self.dq, self.dk, self.dv, self.dom]
        self.inputs = [self.x[n] for n in ("q", "k", "v", "dout", "omega")]

    @staticmethod
    def _ws(n, dev):
        import torch
        return torch.empty(max(256, n), dtype=torch.uint8, device=dev)

    def run(self, stream=None):
        sl, w, x, om = self.slim, self.w, self.x, self.om
        C, f = w.C, w.feature
        if self.mode == "causal":
            sl.forward_into(x["q"], x["k"], x["v"], om, C, f, self.out, self.S, self.z, self.ws_f,
                            stream, S_lo=self.S_lo, z_lo=self.z_lo)
            sl.backward_into(x["q"], x["k"], x["v"], om, self.out, x["dout"], self.S, self.z, C, f,
                             self.dq, self.dk, self.dv, self.dom, self.ws_b, stream,
                             S_lo=self.S_lo, z_lo=self.z_lo)
        elif self.mode == "bidir":
            sl.forward_bidir_into(x["q"], x["k"], x["v"], om, C, f, self.out, self.S, self.z,
                                  self.ws_f, stream)
            sl.backward_bidir_into(x["q"], x["k"], x["v"], om, self.out, x["dout"], self.S,
                                   self.z, C, f, self.dq, self.dk, self.dv, self.dom, self.ws_b,
                                   stream)
        elif self.mode == "stack":
            lib, ls, sx = sl.library(), self.layers, self.sx
            dt, ft = sl.DTYPES[sx["x"].dtype], sl.FEATURES[f]
            B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
            h = sl._stream_handle(stream)
            sl._check(lib.slim_stack_fwd(sx["x"].data_ptr(), sl._ptr(self.soms), B, H, L, d, M, C,
                                         ls, dt, ft, self.y.data_ptr(), self.sS.data_ptr(),
                                         self.sz.data_ptr(), self.sSl.data_ptr(),
                                         self.szl.data_ptr(), self.ws_f.data_ptr(),
                                         self.ws_f.numel(), h), "slim_stack_fwd")
            sl._check(lib.slim_stack_bwd(sx["x"].data_ptr(), sl._ptr(self.soms),
                                         sx["dy"].data_ptr(), self.sS.data_ptr(),
                                         self.sz.data_ptr(), self.sSl.data_ptr(),
                                         self.szl.data_ptr(), B, H, L, d, M, C, ls, dt, ft,
                                         self.dx.data_ptr(),
                                         sl._ptr(self.sdom if self.soms is not None else None),
                                         self.ws_b.data_ptr(), self.ws_b.numel(), h),
                      "slim_stack_bwd")
        else:
            prev = None
            for sg in self.segs:
                sl.forward_into(sg["q"], sg["k"], sg["v"], om, C, f, sg["out"], sg["S"], sg["z"],
                                self.ws_f, stream, S_lo=sg["S_lo"], z_lo=sg["z_lo"],
                                S_init=None if prev is None else prev["S"],
                                z_init=None if prev is None else prev["z"],
                                S_init_lo=None if prev is None else prev["S_lo"],
                                z_init_lo=None if prev is None else prev["z_lo"])
                prev = sg
            nxt = None
            for sg in reversed(self.segs):
                sl.backward_into(sg["q"], sg["k"], sg["v"], om, sg["out"], sg["dout"], sg["S"],
                                 sg["z"], C, f, sg["dq"], sg["dk"], sg["dv"], sg["dom"],
                                 self.ws_b, stream, S_lo=sg["S_lo"], z_lo=sg["z_lo"],
                                 G_S_in=None if nxt is None else nxt["G"],
                                 g_z_in=None if nxt is None else nxt["gz"],
                                 G_S_out=sg["G"], g_z_out=sg["gz"])
                nxt = sg

    def check(self):
        self.slim.check_device_error(self.ws_f)
        self.slim.check_device_error(self.ws_b)


def e2e_pipelined(sets, host_in, host_out, steps, warmup):
    """End to end through the public API: every step copies its inputs in from
    pinned host memory and its results (out, dq, dk, dv, dOmega) back.  Two
    buffer sets alternate, so step i's copy in runs during step i-1's compute
    and its copy out during step i+1's compute, on two copy streams; each step
    still moves its own bytes.  Returns ms for `steps` steps."""
    import torch
    cin, comp, cout = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = {k: [torch.cuda.Event() for _ in range(2)] for k in ("in", "comp", "out")}
    used = [False, False]

    def issue(i):
        b = i % 2
        st = sets[b]
        with torch.cuda.stream(cin):
            if used[b]:
                cin.wait_event(ev["comp"][b])         # step i-2 has read these inputs
            for dst, src in zip(st.inputs, host_in[b]):
                dst.copy_(src, non_blocking=True)
            ev["in"][b].record(cin)
        comp.wait_event(ev["in"][b])
        if used[b]:
            comp.wait_event(ev["out"][b])             # step i-2's results have left
        st.run(comp)
        ev["comp"][b].record(comp)
        with torch.cuda.stream(cout):
            cout.wait_event(ev["comp"][b])
            for dst, src in zip(host_out[b], st.outputs):
                dst.copy_(src, non_blocking=True)
            ev["out"][b].record(cout)
        used[b] = True

    for i in range(warmup):
        issue(i)
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(cin)
    for i in range(warmup, warmup + steps):
        issue(i)
    cout.wait_stream(cin)
    cout.wait_stream(comp)
    t1.record(cout)
    torch.cuda.synchronize()
    return t0.elapsed_time(t1)


def mem_vs_C(dev, steps):
    """Peak device memory and tokens/s for each slice size C of the B2 H8
    L32768 d64 M256 bf16 workload (Sec. 4.1's time/memory-vs-C protocol, Fig. 2):
    workspace bytes, the measured peak above the inputs and outputs (IO floor),
    and the same method on an input of length C alone (the length-C point)."""
    import torch
    from paper_2012_11346_gb300 import slim
    from paper_2012_11346_gb300 import workloads as W
    w0 = W.WORKLOADS["L32768_bf16"]
    x = W.make_inputs(w0, device=dev)
    floor = sum(t.numel() * t.element_size() for t in x.values()) + \
        4 * x["q"].numel() * x["q"].element_size()   # + out, dq, dk, dv
    rows = []
    for C in W.C_SWEEP:
        w = w0.with_(C=C)

        def step():
            o, S, z, Sl, zl = slim.forward(x["q"], x["k"], x["v"], x["omega"], C, w.feature,
                                           residuals=True)
            slim.backward(x["q"], x["k"], x["v"], x["omega"], o, x["dout"], S, z, C, w.feature,
                          S_lo=Sl, z_lo=zl)

        step()
        torch.cuda.synchronize()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(steps):
            step()
        e1.record()
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / steps
        peak = torch.cuda.max_memory_allocated(dev)
        outs = 4 * x["q"].numel() * x["q"].element_size()      # out, dq, dk, dv
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
        rows.append({"C": C, "tokens_per_s": round(w.B * w.L / (ms / 1e3), 1),
                     "ms_per_step": round(ms, 3),
                     "workspace_bytes": slim.workspace_size(w.B, w.H, w.L, w.d, w.M, C,
                                                            x["q"].dtype, w.feature, False)
                     + slim.workspace_size(w.B, w.H, w.L, w.d, w.M, C, x["q"].dtype,
                                           w.feature, True),
                     "peak_above_inputs_bytes": peak - base,
                     "peak_above_io_floor_bytes": peak - base - outs,
                     "length_C_input_above_inputs_bytes": lb_above})
    del x
    torch.cuda.empty_cache()
    return {"workload": "B2 H8 L32768 d64 M256 bf16 exp", "io_floor_bytes": floor,
            "steps_per_C": steps, "rows": rows}


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
    B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
    main = StepSet(w, dev, args.mode, args.segments, layers=args.layers)
    step = main.run

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
    main.check()
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
    main.check()

    # untimed validation pass: every call clears the device error word at its
    # start, so check it after each step; a bounded wait that gave up during
    # the measurement would make the numbers above meaningless
    for _ in range(args.steps):
        step()
        main.check()

    # end to end through the public API: pinned host inputs in, results out,
    # copies overlapped with the neighbouring steps' compute (two buffer sets)
    second = StepSet(w, dev, args.mode, args.segments, x=None, layers=args.layers)
    sets = [main, second]
    host_in = [[t.cpu().pin_memory() for t in st.inputs] for st in sets]
    host_out = [[torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in st.outputs]
                for st in sets]
    h2d = sum(t.numel() * t.element_size() for t in main.inputs)
    d2h = sum(t.numel() * t.element_size() for t in main.outputs)
    barrier(ws)
    ms_e2e = max_over_ranks(e2e_pipelined(sets, host_in, host_out, args.steps, args.warmup), ws)
    e2e_value = tokens / (ms_e2e / 1e3)
    del second, sets, host_in, host_out
    torch.cuda.empty_cache()

    # peak device memory of one fwd+bwd through the allocating API
    peak, base = None, None
    if args.mode == "causal":
        x = main.x
        torch.cuda.synchronize()
        torch.cuda.reset_peak_memory_stats(dev)
        base = torch.cuda.memory_allocated(dev)
        o2, S2, z2, S2l, z2l = slim.forward(x["q"], x["k"], x["v"], main.om, w.C, w.feature,
                                            residuals=True)
        g2 = slim.backward(x["q"], x["k"], x["v"], main.om, o2, x["dout"], S2, z2, w.C,
                           w.feature, S_lo=S2l, z_lo=z2l)
        torch.cuda.synchronize()
        peak = torch.cuda.max_memory_allocated(dev)
        del o2, S2, z2, S2l, z2l, g2

    line = {
        "metric": METRIC, "value": round(value, 1), "unit": "tokens/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms / args.steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": path_dtype(stats, w), "data": "synthetic",
        "config": {"workload": w.name, "B": B, "H": H, "L": L, "d": d, "M": M, "C": w.C,
                   "feature": w.feature, "input_dtype": w.dtype, "mode": args.mode,
                   **({"segments": args.segments} if args.mode == "segments" else {}),
                   **({"layers": args.layers} if args.mode == "stack" else {}),
                   "parallelism": f"replicas x{ws}" if ws > 1 else "single GPU",
                   "l2": "no flush; per-step working set (q,k,v,dout,out,dq,dk,dv) "
                         f"{8 * main.x['q'].numel() * main.x['q'].element_size() / 2**20:.0f} MiB "
                         "> L2 129 MiB"},
        "e2e": {"value": round(e2e_value, 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "overlap": "copies of step i overlap compute of steps i-1 and i+1"},
        "gpu_launches": int(launches),
        "roofline": roofline(stats, args.steps),
        "ceilings": step_ceilings(w, B, H, L, ms / args.steps),
        "profiled_ms_per_step": round(ms_profiled / args.steps, 4),
        "clocks": clocks,
        "peak_mem": ({"bytes": peak, "above_inputs_bytes": peak - base,
                      "workspace_bytes": main.ws_b.numel()} if peak is not None else None),
        "kernels": [{k_: (round(v_, 4) if isinstance(v_, float) else v_) for k_, v_ in s.items()}
                    for s in stats],
    }
    del main
    torch.cuda.empty_cache()
    if (rank == 0 and ws == 1 and not args.no_mem_curve and args.mode == "causal"
            and args.workload == DEFAULT_WORKLOAD and not (args.B or args.H or args.C)):
        line["mem_vs_C"] = mem_vs_C(dev, 3)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        # The oracle pool starts only after every GPU measurement: with an
        # idle pool alive during the GPU passes, the end-to-end pass was
        # measured ~400x slower on a 16-core host.  Spawned workers do not
        # inherit the parent's CUDA context.
        n = oracle_pool_size()
        pool = start_oracle_pool(n)
        tok, sec = oracle_sample(w, {"C": w.C}, pool, n, args.mode, args.layers)
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
            oracle_sample(w, {"C": w.C}, pool, n, args.mode, args.layers)
        tok, sec = 0, 0.0
        for _ in range(args.steps):
            t, s = oracle_sample(w, {"C": w.C}, pool, n, args.mode, args.layers)
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
