"""The tensor-core building blocks (TMA tiles, smem descriptors, TMEM, MMA with
A in tensor memory) against plain matrix products on the same bf16 operands."""
import pytest
import torch

from paper_2601_02819_gb300 import phsa

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed", [0, 1])
def test_selftest_matches_matmul(seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    A = torch.randn((128, 128), generator=g, device="cuda").to(torch.bfloat16)
    B = torch.randn((64, 128), generator=g, device="cuda").to(torch.bfloat16)
    V = torch.randn((64, 128), generator=g, device="cuda").to(torch.bfloat16)
    S, O = phsa.phsa_selftest_tcgen05(A, B, V)
    torch.cuda.synchronize()
    assert phsa.phsa_get_device_status() == 0
    S_ref = A.double() @ B.double().T
    torch.testing.assert_close(S.double(), S_ref, rtol=1e-5, atol=1e-3)
    O_ref = S.to(torch.bfloat16).double() @ V.double()
    torch.testing.assert_close(O.double(), O_ref, rtol=1e-5, atol=1e-3)
