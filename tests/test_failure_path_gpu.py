"""A device-side wait that runs out reports SLIM_ERR_TIMEOUT through the
workspace error word, without faulting: the context keeps working."""
import ctypes

import pytest
import torch

from paper_2012_11346_gb300 import slim
from paper_2012_11346_gb300 import workloads as W

pytestmark = pytest.mark.gpu


def test_bounded_wait_gives_up_and_reports(cuda_device):
    ws = torch.zeros(256, dtype=torch.uint8, device=cuda_device)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    assert slim.library().slim_diag_wait_timeout(ws.data_ptr(), stream) == 0
    with pytest.raises(slim.SlimError) as e:
        slim.check_device_error(ws)
    assert e.value.status == 5                      # SLIM_ERR_TIMEOUT
    slim.check_device_error(ws)                     # the word was cleared
    # the context still runs the real path
    w = W.WORKLOADS["tiny_f32"]
    x = W.make_inputs(w, device=cuda_device)
    out, S, z = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature)
    torch.cuda.synchronize()
    assert torch.isfinite(out).all()


def test_next_call_reports_timeout_without_blocking(cuda_device):
    """A wait that gave up in one call is reported by the next call on the same
    workspace (once the failed kernel has finished), without a blocking read:
    that call returns SLIM_ERR_TIMEOUT and launches nothing; the call after it
    runs normally.  A blocking check that already reported it is not repeated."""
    w = W.WORKLOADS["L4096_bf16"].with_(B=1, H=2, L=600, C=256)
    x = W.make_inputs(w, device=cuda_device)
    need = slim.workspace_size(w.B, w.H, w.L, w.d, w.M, w.C, torch.bfloat16, w.feature, False)
    ws = torch.zeros(need, dtype=torch.uint8, device=cuda_device)
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    ref = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature)
    torch.cuda.synchronize()
    assert slim.library().slim_diag_wait_timeout(ws.data_ptr(), stream) == 0
    torch.cuda.synchronize()                        # the failed kernel has finished
    before = slim.launch_count()
    with pytest.raises(slim.SlimError) as e:
        slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature, workspace=ws)
    assert e.value.status == 5 and slim.launch_count() == before
    out, S, z = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature, workspace=ws)
    torch.cuda.synchronize()
    slim.check_device_error(ws)
    assert torch.equal(out, ref[0]) and torch.equal(S, ref[1])
    # reported by the blocking check first: the next call does not report it again
    assert slim.library().slim_diag_wait_timeout(ws.data_ptr(), stream) == 0
    with pytest.raises(slim.SlimError):
        slim.check_device_error(ws)
    out2, _, _ = slim.forward(x["q"], x["k"], x["v"], x["omega"], w.C, w.feature, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(out2, ref[0])
