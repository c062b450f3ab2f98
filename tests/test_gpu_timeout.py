"""Failure detection of the kernels' bounded waits, driven on the GPU without
a fault: every mbarrier wait gives up after a time limit, records a timeout
that pf_sync_check reports as PF_ERR_TIMEOUT, and the kernel leaves cleanly
(its tensor memory freed, nothing in flight), so the context stays usable.

The test shortens the limit to 2 ms and switches on the GEMM producer's test
hook that issues no operand loads: the MMA warp then waits on a barrier that
nothing will ever complete.  The kernel must return within a few limits, the
timeout must be reported once (and cleared), and the same GEMM run before and
after must give bit-identical results.  A small layer forward and backward
afterwards, whose kernels allocate tensor memory again, must still match the
float64 oracle.
"""
import time

import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.layer import ProxyLayer, to_device
from tests._util import assert_close, assert_grad_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def _gemm(A, B, D, stream):
    M, K = A.shape
    N = B.shape[0]
    pf.pf_gemm_bf16(M, N, K, A, 0, B, 0, D, N, stream)


def test_bounded_wait_runs_out_and_reports_timeout():
    g = torch.Generator(device="cuda").manual_seed(11)
    A = torch.randn(256, 512, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(256, 512, device="cuda", generator=g).to(torch.bfloat16)
    stream = torch.cuda.current_stream().cuda_stream
    D0 = torch.zeros(256, 256, device="cuda")
    _gemm(A, B, D0, stream)
    pf.pf_sync_check(stream)
    ref = (A.double() @ B.double().T).float()
    assert float((D0 - ref).abs().max()) <= 1e-3 * float(ref.abs().max())

    D1 = torch.zeros_like(D0)
    try:
        pf.pf_debug_set_wait_limit_ns(2_000_000)
        pf.pf_debug_gemm_skip_loads(True)
        t0 = time.perf_counter()
        _gemm(A, B, D1, stream)
        with pytest.raises(pf.ProxyFormerError) as e:
            pf.pf_sync_check(stream)
        elapsed = time.perf_counter() - t0
    finally:
        pf.pf_debug_gemm_skip_loads(False)
        pf.pf_debug_set_wait_limit_ns(0)
    assert e.value.status == pf.PF_ERR_TIMEOUT, str(e.value)
    assert "wait ran out" in str(e.value)
    assert elapsed < 5.0, elapsed
    pf.pf_sync_check(stream)  # the flag was cleared by the report

    D2 = torch.zeros_like(D0)
    _gemm(A, B, D2, stream)
    pf.pf_sync_check(stream)
    assert torch.equal(D2, D0)

    spec = S.LayerSpec(batch=1, L=1000, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4)
    inp = S.make_layer_inputs(spec, 12)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.bfloat16)
    G = to_device(inp["G"], torch.bfloat16)
    Xo = lay.forward(X)
    dX = lay.backward(X, G)
    pf.pf_sync_check(stream)
    ref_Xo, _ = OL.layer_fwd(spec, inp, inp["X"])
    ref_dX, _, ref_g = OL.layer_bwd(spec, inp, inp["X"], inp["G"])
    assert_close("X_out", Xo.float().cpu().numpy(), ref_Xo)
    assert_grad_close("dX", dX.float().cpu().numpy(), ref_dX)
    assert_grad_close("grad W_c1", lay.grads["W_c1"].cpu().numpy(), ref_g["W_c1"])
