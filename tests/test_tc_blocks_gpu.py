"""The tensor-core operand layouts (K-major / MN-major, 128-byte swizzle) give
the same product as a plain matrix multiply, for every combination used by the
kernels.  Integer-valued bf16 inputs keep every product and partial sum exact
in fp32, so the comparison is exact."""
import pytest
import torch

from paper_2012_11346_gb300 import slim

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("a_mn", [0, 1])
@pytest.mark.parametrize("b_mn", [0, 1])
@pytest.mark.parametrize("K,N", [(64, 64), (128, 128), (256, 64), (128, 256), (256, 256)])
def test_tc_mma_layouts(cuda_device, a_mn, b_mn, K, N):
    g = torch.Generator(device="cpu").manual_seed(K * 7 + N + 3 * a_mn + b_mn)
    A = torch.randint(-4, 5, (128, K), generator=g).to(torch.bfloat16).to(cuda_device)
    B = torch.randint(-4, 5, (K, N), generator=g).to(torch.bfloat16).to(cuda_device)
    D, err = slim.tc_selftest(A, B, a_mn, b_mn)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    ref = A.float() @ B.float()
    assert torch.equal(D, ref), (D - ref).abs().max().item()
