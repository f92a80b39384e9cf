"""bench.py's step floors: the algorithmic work of one fwd+bwd step (30dM FLOPs,
12ds HBM bytes, 4M exponentials per token-head) and the bound they imply.
Host arithmetic only, no GPU."""
import bench
from paper_2012_11346_gb300 import workloads as W


def test_bench_workload_floors():
    w = W.WORKLOADS["L4096_bf16"]
    c = bench.step_ceilings(w, w.B, w.H, w.L, 1.0)
    th = 8 * 8 * 4096
    assert th == 262144
    assert c["flops"] == 30 * 64 * 256 * th            # 1.29e11
    assert c["hbm_bytes"] == 12 * 64 * 2 * th          # 403 MB
    assert c["exps"] == 4 * 256 * th                   # 2.7e8
    peaks, _ = bench.measured_peaks()
    assert abs(c["floors_us"]["tensor"] - c["flops"] / (peaks["bf16_tflops"] * 1e6)) < 0.01
    assert abs(c["floors_us"]["hbm"] - c["hbm_bytes"] / (peaks["hbm_gbs"] * 1e3)) < 0.01
    assert abs(c["floors_us"]["mufu"] - c["exps"] / bench.MUFU_EX2_PER_S * 1e6) < 0.01
    assert c["bound"] == max(c["floors_us"], key=c["floors_us"].get)
    assert c["t_star_us"] == c["floors_us"][c["bound"]]
    assert abs(c["frac_of_step"] - c["t_star_us"] / 1000.0) < 1e-4


def test_relu_fp32_floors():
    w = W.WORKLOADS["L8192_relu_f32"]
    c = bench.step_ceilings(w, w.B, w.H, w.L, 46.0)
    assert c["exps"] == 0 and c["floors_us"]["mufu"] == 0
    # fp32 products as six bf16-piece products on the tensor pipe
    peaks, _ = bench.measured_peaks()
    assert "tensor x6" in c["floors_us"] and "tensor" not in c["floors_us"]
    assert abs(c["floors_us"]["tensor x6"] - 6 * c["flops"] / (peaks["bf16_tflops"] * 1e6)) < 0.01
    assert c["hbm_bytes"] == 12 * 64 * 4 * w.B * w.H * w.L
