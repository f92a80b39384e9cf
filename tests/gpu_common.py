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


def compare(gpu, ref, tol, names=NAMES, where="", scale=None):
    """rel-L2 per tensor.  A reference that vanishes identically (e.g. dq and
    dk for L = 1, where out_1 = v_1 does not depend on q or k) has no relative
    error; there the error is taken relative to `scale` (the gradient scale,
    e.g. ||dout||) instead."""
    errs = {}
    for n in names:
        g = to64(gpu[n]) if torch.is_tensor(gpu[n]) else np.asarray(gpu[n])
        r = np.asarray(ref[n], dtype=np.float64)
        nr = np.linalg.norm(r.ravel())
        if scale is not None and nr <= 1e-9 * scale:
            errs[n] = float(np.linalg.norm((g - r).ravel()) / scale)
        else:
            errs[n] = oracle.rel_l2(g, r)
    bad = {n: e for n, e in errs.items() if not (e <= tol)}
    assert not bad, f"{where} rel-L2 above {tol}: {bad} (all: {errs})"
    return errs


def cpu_inputs(x):
    return {n: to64(t) for n, t in x.items()}
