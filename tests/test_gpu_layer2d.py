"""2D bidirectional layer (Sec. 3.9) forward + backward on the GPU against
the float64 oracle: patch compression, timestep adaLN on the proxies,
bidirectional proxy attention, decompression with affine injection
(Eq. inj-affine), and every gradient including the timestep MLP's.  Grids
span several GEMM tiles; the largest case has the paper workload's d = 512,
8 x 64 heads, 8 x 8 patches and batch 4 on a 128 x 128 grid."""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.layer import ProxyLayer, to_device
from tests._util import assert_close, assert_grad_close

pytestmark = pytest.mark.gpu


def _spec2d(B, g, d, nh, p):
    return S.LayerSpec(batch=B, L=g * g, d=d, n_heads=nh, P=p * p, mode=S.BIDIR_2D,
                       inject=S.INJ_AFFINE, grid_h=g, grid_w=g, patch=p)


CASES = {
    "g32_d128_p4_b2": (_spec2d(2, 32, 128, 2, 4), True, False),
    "g64_d256_p8": (_spec2d(1, 64, 256, 4, 8), False, False),
    "g128_d512_p8_b4": (_spec2d(4, 128, 512, 8, 8), True, True),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


@pytest.mark.parametrize("name", list(CASES))
def test_layer2d_fwd_bwd_matches_oracle(name):
    spec, with_h_in, strict = CASES[name]
    inp = S.make_layer_inputs(spec, 40 + len(name), with_h_in=with_h_in)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.bfloat16)
    G = to_device(inp["G"], torch.bfloat16)
    t = to_device(inp["t"], torch.float32)
    H_in = to_device(inp["H_in"], torch.float32) if with_h_in else None
    dHo = to_device(inp["dH_out"], torch.float32)
    H_out, dH_in = lay.empty_proxy(), lay.empty_proxy()
    Xo = lay.forward(X, H_in, t, H_out=H_out)
    dX = lay.backward(X, G, H_in, t, dH_out=dHo, dH_in=dH_in)
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    f = lambda a: a.float().cpu().numpy()
    H_in_np = inp.get("H_in")
    ref_Xo, ref_H = OL.layer_fwd(spec, inp, inp["X"], H_in_np, inp["t"])
    ref_dX, ref_dH, ref_g = OL.layer_bwd(spec, inp, inp["X"], inp["G"], H_in_np, inp["t"],
                                         inp["dH_out"])
    (assert_close if strict else assert_grad_close)("X_out", f(Xo), ref_Xo)
    assert_close("H_out", f(H_out), ref_H)
    assert_grad_close("dX", f(dX), ref_dX)
    assert_grad_close("dH_in", f(dH_in), ref_dH)
    for k, v in ref_g.items():
        assert_grad_close("grad " + k, f(lay.grads[k]), v)
