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
