"""A stack of causal 1D layers with layer-wise ratios (Sec. 3.6) against the
float64 oracle composed layer by layer: H is carried between layers with the
same P and re-extracted when P changes; the backward follows the same rule.
Bar, per tensor: twice the bf16 rounding floor of the same problem (the
oracle's equations evaluated again with bf16 rounding at the library's
storage points, test_bf16_error_floor.run_stack), plus 1e-3 on the RMS and
1e-2 on the max error -- rounding compounds through the layers, while a wrong
carry rule moves whole tensors by O(1).  The stack prefill must fill every
layer's proxy KV cache from that layer's own input and proxy stream."""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.stack import ProxyStack
from tests._util import assert_grad_close, max_rel_err, record, rms_rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def _floor_check(name, got, ref, e_ref, e_bf):
    fr, fm = rms_rel_err(e_bf, e_ref), max_rel_err(e_bf, e_ref)
    gr, gm = rms_rel_err(got, ref), max_rel_err(got, ref)
    record(name, got, ref, f"rms {2 * fr + 1e-3:.3g}, max {2 * fm + 1e-2:.3g} (2x floor)")
    assert gr <= 2 * fr + 1e-3 and gm <= 2 * fm + 1e-2, (
        f"{name}: rms {gr:.3e} max {gm:.3e} vs floor rms {fr:.3e} max {fm:.3e}")


def test_stack_matches_composed_oracle():
    from tests.test_bf16_error_floor import ROUNDED, STACK_RATIOS, run_stack, stack_case
    ratios = STACK_RATIOS
    L, d, nh = 1024, 128, 2
    specs = []
    for P in ratios:
        k1, k2 = S.default_factors(P)
        specs.append(S.LayerSpec(batch=1, L=L, d=d, n_heads=nh, P=P, levels=2, k1=k1, k2=k2))
    params = [S.make_layer_params(s, 70 + i) for i, s in enumerate(specs)]
    inp = S.make_layer_inputs(specs[0], 80)
    st = ProxyStack(specs, params)
    X = torch.from_numpy(inp["X"]).cuda().to(torch.bfloat16)
    G = torch.from_numpy(inp["G"]).cuda().to(torch.bfloat16)
    Xo = st.forward(X).float().cpu().numpy()
    dX = st.backward(G).float().cpu().numpy()
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    # oracle: forward layer by layer, keeping each layer's input and H
    xs, hs = [inp["X"].astype(np.float64)], []
    for l, (s, p) in enumerate(zip(specs, params)):
        carry = l > 0 and specs[l].P == specs[l - 1].P
        xo, h = OL.layer_fwd(s, p, xs[-1], hs[-1] if carry else None)
        xs.append(xo)
        hs.append(h)
    g, dh_next, grads = inp["G"].astype(np.float64), None, []
    for l in reversed(range(len(specs))):
        carry = l > 0 and specs[l].P == specs[l - 1].P
        nxt = l + 1 < len(specs) and specs[l + 1].P == specs[l].P
        g, dh_in, gr = OL.layer_bwd(specs[l], params[l], xs[l], g, hs[l - 1] if carry else None,
                                    None, dh_next if nxt else None)
        dh_next = dh_in
        grads.append((l, gr))
    # the bf16 floor of this very problem (same specs, seeds and inputs)
    fspecs, fparams, fX, fG = stack_case()
    assert [f.P for f in fspecs] == list(ratios) and np.array_equal(fX, xs[0][0])
    e_ref = run_stack(fspecs, fparams, fX, fG, set())
    e_bf = run_stack(fspecs, fparams, fX, fG, ROUNDED)
    _floor_check("stack X_out", Xo[0], xs[-1][0], e_ref[0], e_bf[0])
    _floor_check("stack dX", dX[0], g[0], e_ref[1], e_bf[1])
    for l, gr in grads:
        for k in ("W_c1", "W_d1", "W_qkv", "b_g"):
            _floor_check(f"layer {l} grad {k}", st.layers[l].grads[k].cpu().numpy(), gr[k],
                         e_ref[2][l][k], e_bf[2][l][k])


def test_stack_prefill_fills_every_layer_cache():
    """Prefill (Sec. 3.8) through a stack: each layer's cache must equal the
    oracle's bulk prefill of that layer's own input X[l] and incoming proxy
    stream.  Ragged history (partial last block) with two sequences, so the
    carried stream's extra row per sequence is skipped; P changes once."""
    from oracle import decode as OD
    from paper_2608_23463_gb300.decode import ProxyKVCache
    ratios = (16, 16, 32)
    B, L, d, nh = 2, 1000, 128, 2
    specs = []
    for P in ratios:
        k1, k2 = S.default_factors(P)
        specs.append(S.LayerSpec(batch=B, L=L, d=d, n_heads=nh, P=P, levels=2, k1=k1, k2=k2))
    specs[2] = S.LayerSpec(batch=B, L=L, d=d, n_heads=nh, P=32)  # one level
    params = [S.make_layer_params(s, 90 + i) for i, s in enumerate(specs)]
    st = ProxyStack(specs, params)
    dspecs = [S.decode_spec_for_layer(s, L // s.P + 2) for s in specs]
    dprms = [S.decode_params_for_layer(s, p, 95 + i) for i, (s, p) in enumerate(zip(specs, params))]
    caches = [ProxyKVCache(ds, dp, S.make_decode_state(ds, 96, [ds.capacity] * B, [5] * B))
              for ds, dp in zip(dspecs, dprms)]
    X = torch.from_numpy(S.make_layer_inputs(specs[0], 97, with_grads=False)["X"])
    X = X.cuda().to(torch.bfloat16)
    out = st.prefill(X, caches).clone()
    pf.pf_sync_check(torch.cuda.current_stream().cuda_stream)
    # the prefill's forward is the plain inference forward (no atomics: bitwise)
    assert torch.equal(out, st.forward(X, train=False))
    for l, (ds, dp, c) in enumerate(zip(dspecs, dprms, caches)):
        m, r = L // ds.P, L % ds.P
        Xl = st.X[l].float().cpu().numpy()
        H = st.H[l - 1].cpu().numpy() if st.carries(l) else None
        ref = OD.kv_prefill(ds, dp, Xl, H)
        assert c.s["n_proxy"].cpu().numpy().tolist() == [m] * B
        assert c.s["n_open"].cpu().numpy().tolist() == [r] * B
        for k in ("K_proxy", "V_proxy"):
            assert_grad_close(f"layer {l} {k}", c.s[k][:, :m].float().cpu().numpy(), ref[k][:, :m],
                              tol=2e-2, max_tol=1e-1)
        assert np.array_equal(c.s["X_open"][:, :r].float().cpu().numpy(), Xl[:, m * ds.P:])
        for k in ("K_open", "V_open"):
            assert_grad_close(f"layer {l} {k}", c.s[k][:, :r].float().cpu().numpy(), ref[k][:, :r],
                              tol=2e-2, max_tol=1e-1)
