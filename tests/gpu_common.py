"""Helpers shared by the GPU parity tests: run libslim and the oracle on the same
seeded inputs and compare tensor by tensor (rel-L2, the measure of Sec. 4.2)."""
import numpy as np
import torch

import oracle
from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

# rel-L2 bounds per tensor: fp32 inputs, and bf16 inputs with fp32 accumulation
TOL = {"f32": 1e-5, "bf16": 2e-2}
NAMES = ("out", "S_state", "z_state", "dq", "dk", "dv", "domega")


def to64(t):
    return W.as_float64_numpy(t)


def gpu_run(x, C, feature, dout=None):
    """x: dict of device tensors from workloads.make_inputs."""
    out, S, z, S_lo, z_lo = slim.forward(x["q"], x["k"], x["v"], x["omega"], C, feature,
                                         residuals=True)
    dq, dk, dv, dom = slim.backward(x["q"], x["k"], x["v"], x["omega"], out,
                                    x["dout"] if dout is None else dout, S, z, C, feature,
                                    S_lo=S_lo, z_lo=z_lo)
    torch.cuda.synchronize()
    return {"out": out, "S_state": S, "z_state": z, "dq": dq, "dk": dk, "dv": dv, "domega": dom,
            "S_lo": S_lo, "z_lo": z_lo}


def oracle_run(xc, C, feature, dout=None):
    """xc: dict of CPU float64 numpy arrays ([B,H,L,d] and omega)."""
    out, S, z = oracle.oracle_fwd(xc["q"], xc["k"], xc["v"], xc["omega"], C, feature)
    dq, dk, dv, dom, extra = oracle.oracle_bwd(xc["q"], xc["k"], xc["v"], xc["omega"],
                                               xc["dout"] if dout is None else dout, S, z, C,
                                               feature)
    return {"out": out, "S_state": S, "z_state": z, "dq": dq, "dk": dk, "dv": dv, "domega": dom,
            "extra": extra}


SEQ = ("out", "dq", "dk", "dv")  # [B, H, L, d] tensors, checked per slice as well


def _err(g, r, scale, floor=0.0):
    """rel-L2 of g against r; the denominator is at least `floor` (and the
    gradient scale where r vanishes identically)."""
    nr = np.linalg.norm(r.ravel())
    if scale is not None and nr <= 1e-9 * scale:
        return float(np.linalg.norm((g - r).ravel()) / scale)
    if not (np.all(np.isfinite(g)) and np.all(np.isfinite(r))):
        return float("inf")
    return float(np.linalg.norm((g - r).ravel()) / max(nr, floor, 1e-300))


def row_blocks(L, C, tiles=(64, 128)):
    """Row ranges checked on their own: every slice [a, a+b) of C rows (Sec.
    3.2, the last one possibly shorter), and the last tile of each slice at
    each tile height the kernels use (64 rows for the fp32 path, 128 for the
    tensor-core path), which is the ragged one when b is not a multiple."""
    Cs = min(C, L) if L > 0 else 1
    out = []
    for a in range(0, L, Cs):
        b = min(Cs, L - a)
        out.append((f"slice@{a}", a, a + b))
        for T in tiles:
            t0 = a + T * ((b - 1) // T)
            if t0 > a or b < Cs:
                out.append((f"last{T}@{t0}", t0, a + b))
    return out


def compare(gpu, ref, tol, names=NAMES, where="", scale=None, C=None):
    """rel-L2 per tensor.  A reference that vanishes identically (e.g. dq and
    dk for L = 1, where out_1 = v_1 does not depend on q or k) has no relative
    error; there the error is taken relative to `scale` (the gradient scale,
    e.g. ||dout||) instead.

    With C given, the [B, H, L, d] tensors are also checked slice by slice and
    on the last tile of every slice, at the same bound, so that a wrong ragged
    tile is not diluted by the rest.  A block's error is taken relative to its
    own norm, or to the norm a block of its size has at the tensor's RMS value
    if that is larger: the gradient dq = u Omega - q sum(u) cancels, and in a
    block where it happens to be small the bf16 rounding of u (about 2^-9
    relative) stands out against the block's own norm although it is no
    larger than anywhere else.  A wrong or missing tile still gives an error
    of order 1 either way."""
    errs = {}
    for n in names:
        g = to64(gpu[n]) if torch.is_tensor(gpu[n]) else np.asarray(gpu[n])
        r = np.asarray(ref[n], dtype=np.float64)
        errs[n] = _err(g, r, scale)
        if C is not None and n in SEQ and r.ndim == 4:
            rms = np.linalg.norm(r.ravel()) / np.sqrt(max(r.size, 1))
            for tag, a, e in row_blocks(r.shape[2], C):
                gb, rb = g[:, :, a:e], r[:, :, a:e]
                errs[f"{n}[{tag}]"] = _err(gb, rb, scale, floor=rms * np.sqrt(rb.size))
    bad = {n: e for n, e in errs.items() if not (e <= tol)}
    assert not bad, f"{where} rel-L2 above {tol}: {bad} (all: {errs})"
    return errs


def cpu_inputs(x):
    return {n: to64(t) for n, t in x.items()}
