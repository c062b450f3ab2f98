"""The tcgen05 GEMM on its own, through the C ABI (pf_gemm_bf16), against a
float32 product of the same bf16 operands, for every operand layout and for
shapes with ragged M, N and K tails.  Shapes with enough 256 x 256 tiles run
on CTA pairs (M=256 tiles split by rows between the two CTAs); 5000 and 4904
rows leave the second CTA of the last pair with 8 rows and with none."""
import pytest
import torch

import paper_2608_23463_gb300 as pf

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


@pytest.mark.parametrize("M,N,K", [(296, 320, 200), (128, 64, 64), (1024, 2048, 4096),
                                   (4096, 1024, 1024), (2048, 8192, 1024), (5000, 4096, 520),
                                   (4904, 2560, 1000)])
@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 1), (1, 0)])
def test_gemm_layouts(M, N, K, a_mn, b_mn):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N * 3 + K + a_mn * 2 + b_mn)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    Ast = A.t().contiguous() if a_mn else A
    Bst = B.t().contiguous() if b_mn else B
    D = torch.full((M, N), float("nan"), device="cuda")
    pf.pf_gemm_bf16(M, N, K, Ast, a_mn, Bst, b_mn, D, N, torch.cuda.current_stream().cuda_stream)
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    ref = A.double() @ B.double().t()
    err = ((D.double() - ref).abs().max() / ref.pow(2).mean().sqrt()).item()
    assert err < 1e-4, err


def test_gemm_is_deterministic():
    M, N, K = 1024, 1024, 2048
    A = torch.randn(M, K, device="cuda").to(torch.bfloat16)
    B = torch.randn(N, K, device="cuda").to(torch.bfloat16)
    outs = []
    for _ in range(2):
        D = torch.empty(M, N, device="cuda")
        pf.pf_gemm_bf16(M, N, K, A, 0, B, 0, D, N, torch.cuda.current_stream().cuda_stream)
        outs.append(D)
    torch.cuda.synchronize()
    assert torch.equal(outs[0], outs[1])
