"""A sequence cut into two segments, one call pair per segment (streaming):
slim_fwd_from starts the second segment from the state B the first returned
(Sec. 3.2, eq. 16), and slim_bwd_from hands the second segment's G^(0) to the
first segment's backward as its G^(N) (Sec. 3.3, eq. 18).  Together the two
segments must give the one-call result on the whole sequence, and both must
match the oracle run on each segment with the same carries."""
import numpy as np
import pytest
import torch

import oracle
from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

from gpu_common import TOL, compare, cpu_inputs, gpu_run, to64

pytestmark = pytest.mark.gpu

CASES = [
    # workload, split row, expected path
    (W.WORKLOADS["L4096_bf16"].with_(B=2, H=2, L=1000, C=256), 512, 1),   # slice boundary
    (W.WORKLOADS["L4096_bf16"].with_(B=2, H=2, L=1000, C=256), 300, 1),   # inside a slice
    (W.WORKLOADS["L8192_relu_f32"].with_(B=1, H=2, L=700, C=128), 256, 0),
    (W.Workload("f32exp", 1, 2, 300, 32, 48, 64, "f32", "exp", "normal", "iid", seed=4), 128, 0),
    (W.WORKLOADS["L4096_square_bf16"].with_(B=1, H=2, L=600, C=128), 256, 0),
]


def _seg(x, a, b):
    return {n: (t[:, :, a:b].contiguous() if t.dim() == 4 else t) for n, t in x.items()}


@pytest.mark.parametrize("w,a,path", CASES, ids=[f"{c[0].name}-{c[1]}" for c in CASES])
def test_two_segments_equal_one_call(cuda_device, w, a, path):
    assert slim.path_for(w.B, w.H, w.L, w.d, w.M, w.C, W.TORCH_DTYPE[w.dtype], w.feature) == path
    x = W.make_inputs(w, device=cuda_device)
    om = None if w.feature == "square" else x["omega"]
    full = gpu_run(x, w.C, w.feature)
    x1, x2 = _seg(x, 0, a), _seg(x, a, w.L)
    f = w.feature
    o1, S1, z1, S1l, z1l = slim.forward(x1["q"], x1["k"], x1["v"], om, w.C, f, residuals=True)
    o2, S2, z2, S2l, z2l = slim.forward(x2["q"], x2["k"], x2["v"], om, w.C, f, residuals=True,
                                        S_init=S1, z_init=z1, S_init_lo=S1l, z_init_lo=z1l)
    g2 = slim.backward(x2["q"], x2["k"], x2["v"], om, o2, x2["dout"], S2, z2, w.C, f,
                       S_lo=S2l, z_lo=z2l, return_state_grad=True)
    g1 = slim.backward(x1["q"], x1["k"], x1["v"], om, o1, x1["dout"], S1, z1, w.C, f,
                       S_lo=S1l, z_lo=z1l, G_S_in=g2[4], g_z_in=g2[5], return_state_grad=True)
    torch.cuda.synchronize()
    tol = TOL[w.dtype]
    seg = {"out": torch.cat([o1, o2], 2), "S_state": S2, "z_state": z2,
           "dq": torch.cat([g1[0], g2[0]], 2), "dk": torch.cat([g1[1], g2[1]], 2),
           "dv": torch.cat([g1[2], g2[2]], 2)}
    if om is not None:
        seg["domega"] = g1[3] + g2[3]
    # forward across a slice boundary: the same arithmetic as one call
    if a % w.C == 0:
        for n in ("out", "S_state", "z_state"):
            assert torch.equal(seg[n], full[n]), n
    # against the oracle with the same carries
    xc = cpu_inputs(x)
    xc1 = {n: (t[:, :, :a] if t.ndim == 4 else t) for n, t in xc.items()}
    xc2 = {n: (t[:, :, a:] if t.ndim == 4 else t) for n, t in xc.items()}
    r1 = oracle.oracle_fwd(xc1["q"], xc1["k"], xc1["v"], xc1["omega"], w.C, f)
    r2 = oracle.oracle_fwd(xc2["q"], xc2["k"], xc2["v"], xc2["omega"], w.C, f, r1[1], r1[2])
    b2 = oracle.oracle_bwd(xc2["q"], xc2["k"], xc2["v"], xc2["omega"], xc2["dout"], r2[1], r2[2],
                           w.C, f)
    b1 = oracle.oracle_bwd(xc1["q"], xc1["k"], xc1["v"], xc1["omega"], xc1["dout"], r1[1], r1[2],
                           w.C, f, b2[4]["G_S"], b2[4]["g_z"])
    ref = {"out": np.concatenate([r1[0], r2[0]], 2), "S_state": r2[1], "z_state": r2[2],
           "dq": np.concatenate([b1[0], b2[0]], 2), "dk": np.concatenate([b1[1], b2[1]], 2),
           "dv": np.concatenate([b1[2], b2[2]], 2), "domega": b1[3] + b2[3]}
    compare(seg, ref, tol, names=tuple(seg), where=f"two segments at {a}", C=w.C)
    # the state gradient handed between the segments, and G^(0) of the sequence
    for got, want in ((g2[4], b2[4]["G_S"]), (g2[5], b2[4]["g_z"]),
                      (g1[4], b1[4]["G_S"]), (g1[5], b1[4]["g_z"])):
        assert oracle.rel_l2(to64(got), want) <= tol
    # and the one-call run agrees with the segments at the same bound
    for n in seg:
        assert oracle.rel_l2(to64(seg[n]), to64(full[n])) <= tol, n


def test_zero_length_segment_passes_the_state_through(cuda_device):
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=300, C=128)
    x = W.make_inputs(w, device=cuda_device)
    o, S, z = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature)
    e = {n: (t[:, :, :0].contiguous() if t.dim() == 4 else t) for n, t in x.items()}
    o0, S0, z0 = slim.forward(e["q"], e["k"], e["v"], x["omega"], w.C, w.feature, S_init=S, z_init=z)
    G = torch.randn_like(S)
    gz = torch.randn_like(z)
    g = slim.backward(e["q"], e["k"], e["v"], x["omega"], o0, e["dout"], S0, z0, w.C, w.feature,
                      G_S_in=G, g_z_in=gz, return_state_grad=True)
    torch.cuda.synchronize()
    assert torch.equal(S0, S) and torch.equal(z0, z)
    assert torch.equal(g[4], G) and torch.equal(g[5], gz)
    assert torch.count_nonzero(g[3]) == 0
