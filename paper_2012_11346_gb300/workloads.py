"""Seeded synthetic inputs for sliced causal linear attention.

This module draws random numbers and nothing else: it holds none of the
attention arithmetic, so both the CUDA path and the fp64 checker can be fed
from it without sharing any computation.

Every workload draws, from one CPU generator seeded once, in this order:
q, k, v ([B, H, L, d]), Omega ([M, d]) and dout ([B, H, L, d]), all in fp32;
q, k, v and dout are then rounded to the workload's dtype (round to nearest
even for bf16).  Omega stays fp32 (the library takes it in fp32).

Distributions (the paper benchmarks on random input strings, Sec. 4.1; its
per-head width is d = 64, Sec. 4):
  * q, k, v ~ N(0, 1) / d^(1/4), or U(-1, 1) for the ReLU workload;
  * Omega: iid N(0, 1), or orthogonal Gaussian -- each block of d rows is the
    orthonormal factor of the QR decomposition of a d x d Gaussian matrix
    (signs fixed by sign(diag R)), rows then scaled by the norms of fresh
    N(0, I_d) draws (chi(d) lengths), as Performers sample their features;
  * dout ~ N(0, 1).
"""
from dataclasses import dataclass, replace

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    L: int
    d: int
    M: int
    C: int
    dtype: str          # "f32" or "bf16"
    feature: str        # "exp" or "relu"
    qkv_dist: str       # "normal" (N(0,1)/d^0.25) or "uniform" (U(-1,1))
    omega_dist: str     # "iid" or "orthogonal"
    seed: int = 0

    @property
    def chains(self):
        return self.B * self.H

    @property
    def token_heads(self):
        return self.B * self.H * self.L

    def with_(self, **kw):
        return replace(self, **kw)


# The five workloads of the benchmark plan, and the quadratic-map workload.
WORKLOADS = {
    "tiny_f32": Workload("tiny_f32", 1, 1, 256, 16, 32, 64, "f32", "exp", "normal", "iid"),
    "L4096_bf16": Workload("L4096_bf16", 8, 8, 4096, 64, 256, 1024, "bf16", "exp", "normal", "orthogonal"),
    "L32768_bf16": Workload("L32768_bf16", 2, 8, 32768, 64, 256, 1024, "bf16", "exp", "normal", "orthogonal"),
    "L8192_relu_f32": Workload("L8192_relu_f32", 4, 12, 8192, 64, 128, 512, "f32", "relu", "uniform", "iid"),
    "L65536_C16_bf16": Workload("L65536_C16_bf16", 1, 4, 65536, 128, 256, 16, "bf16", "exp", "normal", "orthogonal"),
    # the paper's own experimental feature map (Sec. 4: g(x) = x^2 elementwise,
    # M = d = 64 per head) on the bench shape; Omega is drawn but not used
    "L4096_square_bf16": Workload("L4096_square_bf16", 8, 8, 4096, 64, 64, 1024, "bf16", "square", "normal", "iid"),
}

# Slice sizes swept on the L = 32768 workload (time and peak memory vs C).
C_SWEEP = (64, 256, 1024, 4096, 32768)

TORCH_DTYPE = {"f32": torch.float32, "bf16": torch.bfloat16}


def orthogonal_gaussian(M, d, gen):
    """M x d rows: blocks of d orthonormal rows, each row rescaled to a chi(d)
    length.  A final partial block keeps its first rows."""
    blocks = []
    for _ in range((M + d - 1) // d):
        G = torch.randn(d, d, generator=gen, dtype=torch.float32).double()
        Qf, Rf = torch.linalg.qr(G)
        s = torch.sign(torch.diagonal(Rf))
        s[s == 0] = 1.0
        blocks.append((Qf * s[None, :]).T)        # rows orthonormal
    W = torch.cat(blocks, 0)[:M]
    lengths = torch.randn(M, d, generator=gen, dtype=torch.float32).double().norm(dim=1)
    return (W * lengths[:, None]).float()


def make_inputs(w: Workload, device="cpu"):
    """Returns dict(q, k, v, omega, dout) as torch tensors on `device`.

    q, k, v, dout have dtype TORCH_DTYPE[w.dtype]; omega is fp32."""
    gen = torch.Generator(device="cpu").manual_seed(w.seed)
    shape = (w.B, w.H, w.L, w.d)

    def qkv():
        if w.qkv_dist == "normal":
            return torch.randn(shape, generator=gen, dtype=torch.float32) / (w.d ** 0.25)
        if w.qkv_dist == "uniform":
            return torch.rand(shape, generator=gen, dtype=torch.float32) * 2.0 - 1.0
        raise ValueError(w.qkv_dist)

    q, k, v = qkv(), qkv(), qkv()
    if w.omega_dist == "iid":
        omega = torch.randn(w.M, w.d, generator=gen, dtype=torch.float32)
    elif w.omega_dist == "orthogonal":
        omega = orthogonal_gaussian(w.M, w.d, gen)
    else:
        raise ValueError(w.omega_dist)
    dout = torch.randn(shape, generator=gen, dtype=torch.float32)
    dt = TORCH_DTYPE[w.dtype]
    out = {"q": q.to(dt), "k": k.to(dt), "v": v.to(dt), "omega": omega.contiguous(),
           "dout": dout.to(dt)}
    return {n: t.to(device) for n, t in out.items()}


def as_float64_numpy(t):
    """Exact upcast of a (possibly bf16) tensor to a float64 NumPy array."""
    return t.detach().to("cpu", torch.float64).numpy()


def make_stack_inputs(w: Workload, layers, device="cpu"):
    """Inputs of a stack of `layers` residual layers on workload w's shape:
    dict(x [B,H,L,d], omegas [layers, M, d] fp32, dy [B,H,L,d]).  One generator
    seeded once draws x, then each layer's Omega, then dy, with the workload's
    distributions (x like q)."""
    gen = torch.Generator(device="cpu").manual_seed(w.seed)
    shape = (w.B, w.H, w.L, w.d)
    if w.qkv_dist == "normal":
        x = torch.randn(shape, generator=gen, dtype=torch.float32) / (w.d ** 0.25)
    elif w.qkv_dist == "uniform":
        x = torch.rand(shape, generator=gen, dtype=torch.float32) * 2.0 - 1.0
    else:
        raise ValueError(w.qkv_dist)
    oms = []
    for _ in range(layers):
        if w.omega_dist == "iid":
            oms.append(torch.randn(w.M, w.d, generator=gen, dtype=torch.float32))
        else:
            oms.append(orthogonal_gaussian(w.M, w.d, gen))
    dy = torch.randn(shape, generator=gen, dtype=torch.float32)
    dt = TORCH_DTYPE[w.dtype]
    out = {"x": x.to(dt), "omegas": torch.stack(oms).contiguous(), "dy": dy.to(dt)}
    return {n: t.to(device) for n, t in out.items()}
