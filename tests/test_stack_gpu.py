"""A stack of residual linear-attention layers by Algorithm 1 (slices outer,
layers inner, one state per layer) through the C ABI, against the oracle's
stack (Alg. 1 / Alg. 2 for s layers in fp64) on the same seeded inputs."""
import numpy as np
import pytest
import torch

import oracle
from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

from gpu_common import TOL, compare, to64

pytestmark = pytest.mark.gpu

CASES = [
    # workload, layers
    (W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=700, C=256), 3),       # tensor-core layers
    (W.WORKLOADS["tiny_f32"].with_(B=2, H=1, L=300, C=64), 2),          # fp32 layers
    (W.WORKLOADS["L8192_relu_f32"].with_(B=1, H=2, L=400, C=128, d=32, M=64), 2),
    (W.WORKLOADS["L4096_square_bf16"].with_(B=1, H=2, L=500, C=128), 3),
    (W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=700, C=256), 6),       # deeper, bf16
    (W.WORKLOADS["tiny_f32"].with_(B=1, H=1, L=100, C=32), 64),         # the most layers
]


@pytest.mark.parametrize("w,layers", CASES, ids=[f"{c[0].name}-s{c[1]}" for c in CASES])
def test_stack_matches_oracle(cuda_device, w, layers):
    x = W.make_stack_inputs(w, layers, device=cuda_device)
    oms = None if w.feature == "square" else x["omegas"]
    B, H, L, d = x["x"].shape
    M = x["omegas"].shape[1]
    wf = torch.zeros(slim.stack_workspace_size(B, H, L, d, M, w.C, layers, x["x"].dtype,
                                               w.feature, False), dtype=torch.uint8,
                     device=cuda_device)
    wb = torch.zeros(slim.stack_workspace_size(B, H, L, d, M, w.C, layers, x["x"].dtype,
                                               w.feature, True), dtype=torch.uint8,
                     device=cuda_device)
    y, S, z, Sl, zl = slim.stack_forward(x["x"], oms, w.C, w.feature, layers=layers, workspace=wf)
    dx, dom = slim.stack_backward(x["x"], oms, x["dy"], S, z, w.C, w.feature, S_lo=Sl, z_lo=zl,
                                  workspace=wb)
    torch.cuda.synchronize()
    slim.check_device_error(wf)
    slim.check_device_error(wb)
    xc = to64(x["x"])
    omc = to64(x["omegas"])
    ref_y, ref_S, ref_z = oracle.oracle_stack_fwd(xc, list(omc), w.C, w.feature)
    ref_dx, ref_dom = oracle.oracle_stack_bwd(xc, list(omc), to64(x["dy"]), ref_S, ref_z, w.C,
                                              w.feature)
    got = {"out": y, "S_state": S, "z_state": z, "dq": dx}
    ref = {"out": ref_y, "S_state": ref_S, "z_state": ref_z, "dq": ref_dx}
    if dom is not None:
        got["domega"] = dom
        ref["domega"] = ref_dom
    compare(got, ref, TOL[w.dtype], names=tuple(got), where=f"stack s={layers} {w.name}", C=w.C)


def test_one_layer_stack_is_layer_plus_residual(cuda_device):
    """s = 1: X + Att(u, u, u) with u the normalised rows, against the
    single-layer entry point fed u computed in PyTorch (fp32, rounded to the
    dtype: an element of u may round the other way, hence a tolerance)."""
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=600, C=256)
    x = W.make_stack_inputs(w, 1, device=cuda_device)
    y, S, z = slim.stack_forward(x["x"], x["omegas"], w.C, w.feature, residuals=False)
    xf = x["x"].float()
    u = (xf * w.d ** -0.25 / torch.sqrt((xf * xf).mean(-1, keepdim=True) + 1e-6)).to(x["x"].dtype)
    o, S1, z1 = slim.forward(u, u, u, x["omegas"][0].contiguous(), w.C, w.feature)
    torch.cuda.synchronize()
    ref = xf + o.float()
    assert oracle.rel_l2(to64(y), to64(ref)) < 4e-3
    assert oracle.rel_l2(to64(S[0]), to64(S1)) < 4e-3
    assert oracle.rel_l2(to64(z[0]), to64(z1)) < 4e-3


def test_empty_sequence(cuda_device):
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=0, C=256)
    x = W.make_stack_inputs(w, 2, device=cuda_device)
    y, S, z = slim.stack_forward(x["x"], x["omegas"], w.C, w.feature, residuals=False)
    dx, dom = slim.stack_backward(x["x"], x["omegas"], x["dy"], S, z, w.C, w.feature)
    torch.cuda.synchronize()
    assert y.numel() == 0 and dx.numel() == 0
    assert not S.any() and not z.any() and not dom.any()


@pytest.mark.slow
def test_stack_full_size_sampled_chains(cuda_device):
    """Three layers on the bench workload's shape (B8 H8 L4096 d64 M256 C1024
    bf16), as `bench.py --mode stack --layers 3` runs them: the oracle
    recomputes two chains (chains are independent through every layer; the
    Omegas are shared).  dOmega is checked on a second backward whose dy is
    zero outside the sampled chains (the backward is linear in dy)."""
    w = W.WORKLOADS["L4096_bf16"]
    layers = 3
    x = W.make_stack_inputs(w, layers, device=cuda_device)
    y, S, z, Sl, zl = slim.stack_forward(x["x"], x["omegas"], w.C, w.feature)
    dx, _ = slim.stack_backward(x["x"], x["omegas"], x["dy"], S, z, w.C, w.feature, S_lo=Sl,
                                z_lo=zl)
    keep = [(0, 0), (w.B - 1, w.H - 1)]
    m = torch.zeros_like(x["dy"])
    for b, h in keep:
        m[b, h] = x["dy"][b, h]
    _, dom = slim.stack_backward(x["x"], x["omegas"], m, S, z, w.C, w.feature, S_lo=Sl, z_lo=zl)
    torch.cuda.synchronize()
    omc = list(to64(x["omegas"]))
    ref_dom = 0.0
    for b, h in keep:
        xc = to64(x["x"][b:b + 1, h:h + 1])
        ry, rS, rz = oracle.oracle_stack_fwd(xc, omc, w.C, w.feature)
        rdx, rdom = oracle.oracle_stack_bwd(xc, omc, to64(x["dy"][b:b + 1, h:h + 1]), rS, rz, w.C,
                                            w.feature)
        ref_dom = ref_dom + rdom
        got = {"out": y[b:b + 1, h:h + 1], "S_state": S[:, b:b + 1, h:h + 1],
               "z_state": z[:, b:b + 1, h:h + 1], "dq": dx[b:b + 1, h:h + 1]}
        ref = {"out": ry, "S_state": rS, "z_state": rz, "dq": rdx}
        compare(got, ref, TOL[w.dtype], names=tuple(got), where=f"stack full chain ({b},{h})")
    assert oracle.rel_l2(to64(dom), ref_dom) <= TOL[w.dtype]
