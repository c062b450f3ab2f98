"""The allocation-free backward against the regular one, through the C ABI.

proxy_layer_bwd_noalloc exists for callers that cannot give the library a
workspace: host frameworks whose memory planner owns every device byte, and
latency-critical loops that cannot pay cudaMalloc's device-wide
synchronisation.  It keeps its scratch in a fixed device array inside the
library.  Here the regular proxy_layer_bwd (with a workspace) runs once, then
the allocation-free entry point runs twice in a row -- the second call starts
from whatever the first left in the shared array.  Both run the same
deterministic kernels (fixed reduction orders, no atomics), so each result
must equal the regular one bit for bit.

The file name makes pytest collect it last, so a failure here cannot hide the
results of the other GPU tests in a run that stops at the first failure.
"""
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from paper_2608_23463_gb300.layer import ProxyLayer, to_device

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def test_noalloc_backward_matches_workspace_backward():
    spec = S.LayerSpec(batch=2, L=1000, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4)
    desc = pf.layer_desc(spec)
    assert pf.proxy_layer_workspace_size(desc, 1) <= pf.PF_NOALLOC_SCRATCH_BYTES
    inp = S.make_layer_inputs(spec, 77, with_h_in=True)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.bfloat16)
    G = to_device(inp["G"], torch.bfloat16)
    H_in = to_device(inp["H_in"], torch.float32)
    dHo = to_device(inp["dH_out"], torch.float32)
    stream = torch.cuda.current_stream().cuda_stream
    lay.forward(X, H_in)
    dH_ref = lay.empty_proxy()
    dX_ref = lay.backward(X, G, H_in, dH_out=dHo, dH_in=dH_ref)
    pf.pf_sync_check(stream)
    ref = {"dX": dX_ref.clone(), "dH_in": dH_ref.clone()}
    ref.update({k: v.clone() for k, v in lay.grads.items()})

    for call in range(2):
        dX = torch.full_like(dX_ref, float("nan"))
        dH = torch.full_like(dH_ref, float("nan"))
        grads = {k: torch.full_like(v, float("nan")) for k, v in lay.grads.items()}
        pf.proxy_layer_bwd_noalloc(lay.desc, lay.p_struct, X, H_in, None, lay.saved, G, dHo, dX,
                                   dH, pf.layer_params(grads, grads=True), stream)
        pf.pf_sync_check(stream)
        got = {"dX": dX, "dH_in": dH}
        got.update(grads)
        for k in ref:
            assert torch.equal(got[k], ref[k]), f"call {call}: {k} differs from proxy_layer_bwd"


def test_noalloc_rejects_layers_beyond_its_scratch():
    spec = S.LayerSpec(batch=1, L=65536, d=1024, n_heads=16, P=64)
    desc = pf.layer_desc(spec)
    assert pf.proxy_layer_workspace_size(desc, 1) > pf.PF_NOALLOC_SCRATCH_BYTES
    dummy = pf.layer_params({})
    with pytest.raises(pf.ProxyFormerError) as e:
        pf.proxy_layer_bwd_noalloc(desc, dummy, 4096, None, None, 4096, 4096, None, 4096, None,
                                   pf.layer_params({}, grads=True))
    assert e.value.status == pf.PF_ERR_WORKSPACE
    assert "scratch" in str(e.value)
