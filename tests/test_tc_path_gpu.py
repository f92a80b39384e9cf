"""Parity of the tensor-core (tcgen05) path with the oracle: bf16 inputs,
d = 64, M in {128, 256}, both feature maps, full and ragged tiles and slices.
Every case asserts first that the tensor-core kernels are the ones serving it."""
import pytest
import torch

from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

from gpu_common import TOL, compare, cpu_inputs, gpu_run, oracle_run, to64

pytestmark = pytest.mark.gpu


def test_path_selection():
    assert slim.path_for(8, 8, 4096, 64, 256, 1024, torch.bfloat16, "exp") == 1
    assert slim.path_for(2, 8, 32768, 64, 256, 64, torch.bfloat16, "exp") == 1
    assert slim.path_for(4, 12, 8192, 64, 128, 512, torch.float32, "relu") == 0
    assert slim.path_for(1, 4, 65536, 128, 256, 16, torch.bfloat16, "exp") == 0


CASES = [
    # (M, L, C, feature)
    (256, 128, 128, "exp"),      # one full tile
    (256, 1000, 256, "exp"),     # 2-tile slices, ragged last slice and tile
    (256, 777, 128, "relu"),
    (128, 640, 512, "exp"),
    (128, 300, 64, "relu"),      # 64-row slices (half-filled tiles)
    (256, 513, 4096, "exp"),     # C > L
    (256, 1000, 200, "exp"),     # slices of 128 + 72 rows: a ragged tile in every slice
    (128, 700, 320, "relu"),     # 3-tile slices (128 + 128 + 64), ragged last slice
]


@pytest.mark.parametrize("M,L,C,feature", CASES)
def test_tc_parity(cuda_device, M, L, C, feature):
    w = W.Workload("tc", 2, 2, L, 64, M, C, "bf16", feature,
                   "uniform" if feature == "relu" else "normal", "orthogonal", seed=11)
    assert slim.path_for(w.B, w.H, L, 64, M, C, torch.bfloat16, feature) == 1
    x = W.make_inputs(w, device=cuda_device)
    compare(gpu_run(x, C, feature), oracle_run(cpu_inputs(x), C, feature), TOL["bf16"],
            where=f"tc M{M} L{L} C{C} {feature}", C=C)


def test_tc_matches_fp32_path(cuda_device, monkeypatch):
    """The same bf16 problem through both paths: they agree within the bf16
    tolerance (the fp32 path keeps fp32 operands)."""
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=1536)
    x = W.make_inputs(w, device=cuda_device)
    a = gpu_run(x, w.C, w.feature)
    monkeypatch.setenv("SLIM_PATH", "simt")
    assert slim.path_for(1, 2, 1536, 64, 256, w.C, torch.bfloat16, "exp") == 0
    b = gpu_run(x, w.C, w.feature)
    import oracle
    for n in ("out", "S_state", "z_state", "dq", "dk", "dv", "domega"):
        assert oracle.rel_l2(to64(a[n]), to64(b[n])) <= TOL["bf16"], n


def _run_case(cuda_device, B, H, L, C, seed=3, M=256):
    w = W.Workload("tc", B, H, L, 64, M, C, "bf16", "exp", "normal", "orthogonal", seed=seed)
    assert slim.path_for(B, H, L, 64, M, C, torch.bfloat16, "exp") == 1
    x = W.make_inputs(w, device=cuda_device)
    compare(gpu_run(x, C, "exp"), oracle_run(cpu_inputs(x), C, "exp"), TOL["bf16"],
            where=f"tc B{B} H{H} L{L} C{C}")


def test_tc_single_long_chain(cuda_device):
    """One chain of 64 tiles (8 slices of 8): every prefix is handed along a
    single chain, in the forward and in both backward chains."""
    _run_case(cuda_device, 1, 1, 8192, 1024)


def test_tc_many_short_chains(cuda_device):
    """256 chains of 2 tiles, one tile per slice: hand-offs across slice
    boundaries only."""
    _run_case(cuda_device, 16, 16, 256, 128)


def _ring(B, H, L, C, M):
    return slim.bwd_schedule(B, H, L, 64, M, C, torch.bfloat16, "exp")[1]


def test_tc_handoff_ring_wraps_short_stages(cuda_device):
    """Two chains of one-tile slices: stages of 2 items, so the running-sum
    flag is polled just before the adds, and the 16-slot hand-off ring is
    reused over 32 slices (each tile of slice n waits for slice n+16's tile at
    its position to have read its slot)."""
    assert _ring(1, 2, 4096, 128, 256) == 16
    _run_case(cuda_device, 1, 2, 4096, 128)


def test_tc_handoff_ring_wraps_long_stages(cuda_device):
    """128 chains of one-tile slices of 64 rows: stages of 128 items, so the
    running-sum flag is polled up front, and the 4-slot ring is reused (5
    slices)."""
    assert _ring(4, 32, 320, 64, 128) == 4
    _run_case(cuda_device, 4, 32, 320, 64, M=128)


def test_tc_workspace_reuse(cuda_device):
    """Back-to-back calls on one workspace give identical results: the chain
    flags and tile counters start afresh in every call."""
    w = W.Workload("tc", 2, 4, 1536, 64, 256, 512, "bf16", "exp", "normal", "orthogonal", seed=9)
    x = W.make_inputs(w, device=cuda_device)
    q, k, v, om, dout = x["q"], x["k"], x["v"], x["omega"], x["dout"]
    B, H, L, d, M = w.B, w.H, w.L, w.d, w.M
    wsf = torch.empty(slim.workspace_size(B, H, L, d, M, w.C, q.dtype, "exp", False),
                      dtype=torch.uint8, device=cuda_device)
    wsb = torch.empty(slim.workspace_size(B, H, L, d, M, w.C, q.dtype, "exp", True),
                      dtype=torch.uint8, device=cuda_device)
    runs = []
    for _ in range(3):
        out, S, z = slim.forward(q, k, v, om, w.C, "exp", workspace=wsf)
        g = slim.backward(q, k, v, om, out, dout, S, z, w.C, "exp", workspace=wsb)
        torch.cuda.synchronize()
        slim.check_device_error(wsf)
        slim.check_device_error(wsb)
        runs.append([out, S, z, *g])
    for a, b in zip(runs[0], runs[2]):
        assert torch.equal(a, b)
