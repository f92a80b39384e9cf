"""The seeded input generator: determinism, dtype rounding, Omega structure."""
import numpy as np
import torch

from paper_2012_11346_gb300 import workloads as W


def test_deterministic_and_seeded():
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=64)
    a, b = W.make_inputs(w), W.make_inputs(w)
    c = W.make_inputs(w.with_(seed=1))
    for n in a:
        assert torch.equal(a[n], b[n])
        assert not torch.equal(a[n], c[n])


def test_shapes_and_dtypes():
    for w in W.WORKLOADS.values():
        s = w.with_(B=1, H=1, L=32)
        x = W.make_inputs(s)
        for n in ("q", "k", "v", "dout"):
            assert x[n].shape == (1, 1, 32, w.d)
            assert x[n].dtype == W.TORCH_DTYPE[w.dtype]
        assert x["omega"].shape == (w.M, w.d) and x["omega"].dtype == torch.float32


def test_bf16_is_round_to_nearest_even_of_fp32_draw():
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=1, L=128)
    x32 = W.make_inputs(w.with_(dtype="f32"))
    x16 = W.make_inputs(w)
    for n in ("q", "k", "v", "dout"):
        # independent RNE: add the rounding bias to the fp32 bit pattern
        bits = x32[n].view(torch.int32).to(torch.int64) & 0xFFFFFFFF
        lsb = (bits >> 16) & 1
        rounded = ((bits + 0x7FFF + lsb) >> 16) << 16
        rounded = rounded.to(torch.int64)
        rounded = torch.where(rounded >= 2 ** 31, rounded - 2 ** 32, rounded).to(torch.int32)
        assert torch.equal(rounded.view(torch.float32), x16[n].float())


def test_orthogonal_omega_blocks():
    gen = torch.Generator().manual_seed(3)
    d, M = 16, 40
    Om = W.orthogonal_gaussian(M, d, gen).double().numpy()
    dirs = Om / np.linalg.norm(Om, axis=1, keepdims=True)
    for b0 in range(0, M, d):
        blk = dirs[b0:b0 + d]
        G = blk @ blk.T
        assert np.allclose(G, np.eye(len(blk)), atol=1e-6)
    # chi(d) lengths: mean close to sqrt(d - 1/2)
    gen = torch.Generator().manual_seed(4)
    lengths = np.linalg.norm(W.orthogonal_gaussian(4096, d, gen).double().numpy(), axis=1)
    assert abs(lengths.mean() - np.sqrt(d - 0.5)) < 0.05


def test_qkv_distributions():
    w = W.WORKLOADS["L4096_bf16"].with_(B=2, H=2, L=2048, dtype="f32")
    x = W.make_inputs(w)
    assert abs(x["q"].std().item() - w.d ** -0.25) < 0.01
    u = W.make_inputs(W.WORKLOADS["L8192_relu_f32"].with_(B=1, H=1, L=4096))
    assert u["q"].min() >= -1 and u["q"].max() <= 1 and abs(u["q"].mean().item()) < 0.02
