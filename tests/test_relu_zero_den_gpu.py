"""ReLU rows whose denominator is exactly zero, on both CUDA paths.

The feature map must be positive for eq. 2's division to be defined (Sec.
2.1).  The generalized-ReLU map is zero wherever omega_m . q <= 0, so a query
with omega_m . q < 0 for every m has g(q) = 0 and a zero denominator.  The
reading adopted for that row: output 0 and no gradient through it.  Here
column 0 of Omega is made positive and a few query rows are -e_0, so that
omega_m . q = -omega_m0 < 0 exactly (also for Omega rounded to bf16).  The
rows sit in the first tile, a middle tile and the ragged last tile.
"""
import numpy as np
import pytest
import torch

from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

from gpu_common import TOL, compare, cpu_inputs, gpu_run, oracle_run

pytestmark = pytest.mark.gpu

ZERO_ROWS = (0, 200, 517)


def _inputs(w, dev):
    x = W.make_inputs(w, device="cpu")
    om = x["omega"].clone()
    om[:, 0] = om[:, 0].abs() + 0.25
    x["omega"] = om
    q = x["q"].clone()
    for r in ZERO_ROWS:
        q[:, :, r] = 0
        q[:, :, r, 0] = -1
    x["q"] = q
    return {n: t.to(dev) for n, t in x.items()}


@pytest.mark.parametrize("dtype,path", [("bf16", 1), ("f32", 0)], ids=["tensor_core", "fp32"])
def test_relu_zero_denominator_rows(cuda_device, dtype, path):
    w = W.Workload("relu0", 2, 2, 600, 64, 128, 256, dtype, "relu", "uniform", "iid", seed=21)
    assert slim.path_for(w.B, w.H, w.L, w.d, w.M, w.C, W.TORCH_DTYPE[dtype], "relu") == path
    x = _inputs(w, cuda_device)
    xc = cpu_inputs(x)
    ref = oracle_run(xc, w.C, "relu")
    for r in ZERO_ROWS:     # the oracle's reading: zero output, zero query gradient
        assert np.all(ref["out"][:, :, r] == 0) and np.all(ref["dq"][:, :, r] == 0)
    g = gpu_run(x, w.C, "relu")
    for r in ZERO_ROWS:
        assert torch.count_nonzero(g["out"][:, :, r]) == 0, r
        assert torch.count_nonzero(g["dq"][:, :, r]) == 0, r
    for n in ("out", "dq", "dk", "dv", "domega"):
        assert torch.isfinite(g[n]).all(), n
    compare(g, ref, TOL[dtype], where=f"relu zero-den {dtype}", C=w.C)
