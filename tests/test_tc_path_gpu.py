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
]


@pytest.mark.parametrize("M,L,C,feature", CASES)
def test_tc_parity(cuda_device, M, L, C, feature):
    w = W.Workload("tc", 2, 2, L, 64, M, C, "bf16", feature,
                   "uniform" if feature == "relu" else "normal", "orthogonal", seed=11)
    assert slim.path_for(w.B, w.H, L, 64, M, C, torch.bfloat16, feature) == 1
    x = W.make_inputs(w, device=cuda_device)
    compare(gpu_run(x, C, feature), oracle_run(cpu_inputs(x), C, feature), TOL["bf16"],
            where=f"tc M{M} L{L} C{C} {feature}")


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
