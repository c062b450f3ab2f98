"""The layer with temporal-distance ratios (Sec. 3.6) on the GPU against the
float64 oracle: coarse blocks for distant history, finer ones for recent
tokens, one causal attention over all proxies.  Cases: two segments with one
level and a ragged last segment, three segments with two levels, and a single
segment, which must match the ordinary layer's result on the same weights."""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.layer import ProxyLayer
from paper_2608_23463_gb300.segments import ProxySegmentLayer
from tests._util import assert_grad_close

pytestmark = pytest.mark.gpu

CASES = {
    "two_segments_1lvl_ragged": (1, [(512, 32), (250, 8)], S.INJ_GATED),
    "three_segments_2lvl": (2, [(1024, 64, 8, 8), (512, 16, 4, 4), (262, 4, 2, 2)], S.INJ_GATED),
    "two_segments_add": (1, [(256, 16), (256, 16)], S.INJ_ADD),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def _np(t):
    return t.float().cpu().numpy()


@pytest.mark.parametrize("name", list(CASES))
def test_segments_match_oracle(name):
    levels, segs, inject = CASES[name]
    d, nh = 128, 2
    L = sum(s[0] for s in segs)
    kw = dict(k1=segs[0][2], k2=segs[0][3]) if levels == 2 else {}
    spec = S.LayerSpec(batch=1, L=L, d=d, n_heads=nh, P=segs[0][1], levels=levels, inject=inject,
                       **kw)
    shared, seg_prm = S.make_segment_params(d, nh, levels, segs, 80)
    if inject == S.INJ_ADD:
        shared = {k: v for k, v in shared.items() if k not in ("w_x", "w_dlt", "b_g")}
    rng = np.random.default_rng(81)
    X = S.round_bf16(rng.standard_normal((L, d)).astype(np.float32))
    G = S.round_bf16(rng.standard_normal((L, d)).astype(np.float32))
    lay = ProxySegmentLayer(spec, segs, shared, seg_prm)
    Xd = torch.from_numpy(X).cuda().to(torch.bfloat16)[None]
    Xo = lay.forward(Xd)
    dX = lay.backward(Xd, torch.from_numpy(G).cuda().to(torch.bfloat16)[None])
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    f64 = lambda p: {k: v.astype(np.float64) for k, v in p.items()}
    sh64, sp64 = f64(shared), [f64(p) for p in seg_prm]
    if inject == S.INJ_ADD:  # the oracle's gate with zero weights and a huge bias is addition
        sh64.update(w_x=np.zeros(d), w_dlt=np.zeros(d), b_g=np.full(d, 60.0))
    ref_Xo, _ = OL.layer_fwd_segments(spec, segs, sp64, sh64, X)
    ref_dX, ref_sg, ref_g = OL.layer_bwd_segments(spec, segs, sp64, sh64, X, G)
    assert_grad_close("X_out", _np(Xo[0]), ref_Xo)
    assert_grad_close("dX", _np(dX[0]), ref_dX)
    for k in shared:
        assert_grad_close("grad " + k, lay.grads[k].cpu().numpy(), ref_g[k])
    for i, sg in enumerate(ref_sg):
        for k in seg_prm[i]:
            assert_grad_close(f"segment {i} grad {k}", lay.seg_grads[i][k].cpu().numpy(), sg[k])


def test_one_segment_is_the_ordinary_layer():
    """One segment runs the same kernels as the ordinary layer: outputs and
    gradients equal on the same weights (ragged tail, two levels)."""
    spec = S.LayerSpec(batch=1, L=1000, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4)
    inp = S.make_layer_inputs(spec, 82, with_grads=True)
    prm = {k: v for k, v in inp.items() if k.startswith(("W_", "w_", "b_"))}
    seg = {k: v for k, v in prm.items() if k in S.SEGMENT_KEYS}
    shared = {k: v for k, v in prm.items() if k not in S.SEGMENT_KEYS}
    X = torch.from_numpy(inp["X"]).cuda().to(torch.bfloat16)
    G = torch.from_numpy(inp["G"]).cuda().to(torch.bfloat16)
    a = ProxySegmentLayer(spec, [(1000, 16, 4, 4)], shared, [seg])
    b = ProxyLayer(spec, inp)
    xa, xb = a.forward(X), b.forward(X)
    da, db = a.backward(X, G), b.backward(X, G)
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    assert torch.equal(xa, xb)
    assert torch.equal(da, db)
    for k in seg:
        assert torch.equal(a.seg_grads[0][k], b.grads[k]), k
