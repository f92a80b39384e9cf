"""slim_fwd_noalloc: the forward for callers that cannot allocate device
memory (it runs in a scratch array the library reserves up front).  Called
through the C ABI with caller-owned inputs and outputs, twice in a row (the
second call finds the first call's leftovers in the shared scratch), and
checked against slim_fwd, the entry point with a caller workspace.

Collected last on purpose, so a run that stops at the first failure has run
everything else first."""
import ctypes

import pytest
import torch

from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

pytestmark = pytest.mark.gpu

SCRATCH_BYTES = 16 * 1024 * 1024


def _noalloc(x, w, outs):
    out, S, z, S_lo, z_lo = outs
    st = slim.library().slim_fwd_noalloc(
        x["q"].data_ptr(), x["k"].data_ptr(), x["v"].data_ptr(), x["omega"].data_ptr(),
        w.B, w.H, w.L, w.d, w.M, w.C, slim.DTYPES[x["q"].dtype], slim.FEATURES[w.feature],
        out.data_ptr(), S.data_ptr(), z.data_ptr(), S_lo.data_ptr(), z_lo.data_ptr(),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    return st


def _outputs(w, dev, dt):
    return (torch.empty(w.B, w.H, w.L, w.d, dtype=dt, device=dev),
            torch.empty(w.B, w.H, w.M, w.d, dtype=torch.float32, device=dev),
            torch.empty(w.B, w.H, w.M, dtype=torch.float32, device=dev),
            torch.empty(w.B, w.H, w.M, w.d, dtype=torch.float32, device=dev),
            torch.empty(w.B, w.H, w.M, dtype=torch.float32, device=dev))


@pytest.mark.parametrize("w", [
    W.WORKLOADS["L4096_bf16"].with_(B=2, H=4, L=1000, C=256),     # tensor-core kernels
    W.WORKLOADS["tiny_f32"].with_(B=2, H=2, L=300, C=64),         # fp32 kernels
], ids=["bf16_tc", "f32"])
def test_noalloc_matches_slim_fwd_twice(cuda_device, w):
    x = W.make_inputs(w, device=cuda_device)
    ref = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature, residuals=True)
    torch.cuda.synchronize()
    for call in range(2):
        outs = _outputs(w, cuda_device, x["q"].dtype)
        assert _noalloc(x, w, outs) == 0, f"call {call}"
        torch.cuda.synchronize()
        for name, got, want in zip(("out", "S_state", "z_state", "S_lo", "z_lo"), outs, ref):
            assert torch.equal(got, want), (call, name)


def test_noalloc_rejects_problems_beyond_its_scratch(cuda_device):
    w = W.WORKLOADS["L4096_bf16"]   # B8 H8 L4096 C1024 needs ~43 MB of scratch
    need = slim.workspace_size(w.B, w.H, w.L, w.d, w.M, w.C, torch.bfloat16, w.feature, False)
    assert need > SCRATCH_BYTES
    x = W.make_inputs(w.with_(L=w.L), device=cuda_device)
    outs = _outputs(w, cuda_device, torch.bfloat16)
    assert _noalloc(x, w, outs) == 3  # SLIM_ERR_WORKSPACE
