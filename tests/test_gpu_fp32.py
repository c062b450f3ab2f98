"""fp32 layer forward (CUDA cores) against the float64 oracle: the paper-size
fp32 workload (L = 4096, d = 256, 4 x 64 heads, P = 64) and smaller ragged,
batched, two-level and bidirectional variants.  Bar: max|gpu - oracle| <=
1e-4 * RMS(oracle) on X_out, H_out and the injected update X_out - X."""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.layer import ProxyLayer, to_device
from tests._util import F32_TOL, assert_close

pytestmark = pytest.mark.gpu

CASES = {
    "paper_fp32": (S.spec_c1(), False),
    "ragged_b2_2lvl": (S.LayerSpec(batch=2, L=1000, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4,
                                   dtype=S.F32), True),
    "bidir_add": (S.LayerSpec(batch=1, L=512, d=64, n_heads=1, P=8, mode=S.BIDIR_1D,
                              inject=S.INJ_ADD, dtype=S.F32), True),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


@pytest.mark.parametrize("name", list(CASES))
def test_fp32_forward_matches_oracle(name):
    spec, with_h_in = CASES[name]
    inp = S.make_layer_inputs(spec, 0, with_h_in=with_h_in, with_grads=False)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.float32)
    H_in = to_device(inp["H_in"], torch.float32) if with_h_in else None
    H_out = lay.empty_proxy()
    Xo = lay.forward(X, H_in, H_out=H_out)
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    ref_Xo, ref_H = OL.layer_fwd(spec, inp, inp["X"], inp.get("H_in"))
    got = Xo.cpu().numpy()
    assert_close("X_out", got, ref_Xo, F32_TOL)
    assert_close("X_out - X", got - inp["X"], ref_Xo - inp["X"], F32_TOL)
    assert_close("H_out", H_out.cpu().numpy(), ref_H, F32_TOL)


def test_fp32_backward_is_rejected():
    spec = S.spec_c1()
    inp = S.make_layer_inputs(spec, 0, with_grads=True)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.float32)
    with pytest.raises(pf.ProxyFormerError) as e:
        lay.backward(X, X)
    assert e.value.status == pf.PF_ERR_UNSUPPORTED
