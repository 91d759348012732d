"""The tcgen05 bf16 GEMM (the contraction of the workers' dense layers)
against a plain fp32 product of the same bf16 operands."""
import pytest
import torch

import paper_2102_08550_gb300 as P

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("M,N,K", [
    (128, 64, 64),      # one tile, one K-block
    (128, 128, 128),
    (256, 96, 200),     # ragged N and a ragged K tail (200 = 3*64 + 8)
    (512, 784, 64),     # weight-gradient shape of the 784-512 layer
    (384, 128, 784),    # forward shape, 13 K-blocks
    (128, 300, 1024),   # deep K pipeline, ragged N
])
def test_gemm_matches_fp32_product(cuda_device, M, N, K):
    g = torch.Generator(device="cpu").manual_seed(M * 7 + N * 3 + K)
    A = torch.randn(M, K, generator=g).to(torch.bfloat16).to(cuda_device)
    B = torch.randn(N, K, generator=g).to(torch.bfloat16).to(cuda_device)
    C = torch.full((M, N), float("nan"), device=cuda_device)
    P.oscars_gemm_bf16_nt(A.data_ptr(), B.data_ptr(), C.data_ptr(), M, N, K,
                          torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    ref = A.double() @ B.double().T
    err = (C.double() - ref).abs().max().item()
    assert torch.isfinite(C).all()
    assert err <= 1e-5 * ref.abs().max().item() + 1e-6, err


def test_gemm_rejects_bad_shapes(cuda_device):
    A = torch.zeros(100, 64, dtype=torch.bfloat16, device=cuda_device)
    C = torch.zeros(100, 64, device=cuda_device)
    with pytest.raises(P.OscarsError):
        P.oscars_gemm_bf16_nt(A.data_ptr(), A.data_ptr(), C.data_ptr(), 100, 64, 64)
