"""Layer forward + backward on the GPU against the float64 oracle, on seeded
inputs from pf_synth.  Shapes span several GEMM and attention tiles and include
ragged tails (L % P != 0), batches, L < P, both cascade depths and both 1D
modes; the widest cases are the paper-size layers (d = 1024, 16 heads,
P = 64 single-level and 8x8) at a shorter L.  The gated cross-attention
injection runs through the same test, including the cases where some or all
tokens see no proxy.  Bit-exact checks: determinism,
causality perturbation and the block-routing probe."""
import numpy as np
import pytest
import torch

import paper_2608_23463_gb300 as pf
import pf_synth as S
from oracle import layer as OL
from paper_2608_23463_gb300.layer import ProxyLayer, to_device
from tests._util import (CROSS_MAX_TOL, CROSS_TOL, assert_close, assert_grad_close,
                         assert_update_close)

pytestmark = pytest.mark.gpu

# name: (spec, with_h_in, strict).  strict: the forward output X_out is held to
# max|err| <= 2e-2 RMS (the paper-shaped d = 1024 layers); the small synthetic
# variants (d <= 128, add injection) use the RMS bar, since their bf16 floor
# is above 2e-2 max (see test_bf16_error_floor.py).
CASES = {
    "causal_gated_1lvl_b2": (S.LayerSpec(batch=2, L=4000, d=128, n_heads=2, P=16), True, False),
    "causal_gated_2lvl_ragged": (S.LayerSpec(batch=1, L=4136, d=128, n_heads=2, P=16, levels=2,
                                             k1=4, k2=4), True, False),
    "causal_gated_1lvl_ragged_b2": (S.LayerSpec(batch=2, L=1000, d=128, n_heads=2, P=24),
                                    False, False),
    "bidir_add_2lvl_b2": (S.LayerSpec(batch=2, L=2048, d=64, n_heads=1, P=8, levels=2, k1=4,
                                      k2=2, mode=S.BIDIR_1D, inject=S.INJ_ADD), False, False),
    "L_lt_P_b3": (S.LayerSpec(batch=3, L=40, d=128, n_heads=2, P=64), False, False),
    "d1024_P64": (S.LayerSpec(batch=1, L=8192, d=1024, n_heads=16, P=64), False, True),
    "d1024_P64_8x8": (S.LayerSpec(batch=1, L=16384, d=1024, n_heads=16, P=64, levels=2, k1=8,
                                  k2=8), True, True),
    # 9728 rows of 8192: enough rows per CTA for the streaming injection backward
    "d1024_P64_8x8_L77824": (S.LayerSpec(batch=1, L=77824, d=1024, n_heads=16, P=64, levels=2,
                                         k1=8, k2=8), False, True),
    # gated cross-attention injection (Eq. inj-cross): ragged with two
    # sequences (direct dX per sequence), bidirectional, P = 256 (query tiles
    # that see no proxy), L < P (no token sees a proxy), the paper width
    "cross_causal_1lvl_ragged_b2": (S.LayerSpec(batch=2, L=1990, d=128, n_heads=2, P=16,
                                                inject=S.INJ_CROSS), True, False),
    "cross_causal_2lvl_P64_ragged": (S.LayerSpec(batch=1, L=4136, d=128, n_heads=2, P=64,
                                                 levels=2, k1=8, k2=8, inject=S.INJ_CROSS),
                                     True, False),
    "cross_bidir_1lvl_b2": (S.LayerSpec(batch=2, L=1024, d=128, n_heads=2, P=16,
                                        mode=S.BIDIR_1D, inject=S.INJ_CROSS), False, False),
    "cross_causal_P256": (S.LayerSpec(batch=1, L=2048, d=128, n_heads=2, P=256, levels=2,
                                      k1=16, k2=16, inject=S.INJ_CROSS), False, False),
    "cross_L_lt_P_b2": (S.LayerSpec(batch=2, L=40, d=128, n_heads=2, P=64, inject=S.INJ_CROSS),
                        False, False),
    "cross_d1024_P64_8x8": (S.LayerSpec(batch=1, L=4096, d=1024, n_heads=16, P=64, levels=2,
                                        k1=8, k2=8, inject=S.INJ_CROSS), True, True),
    # asymmetric widths (the language model's history stream, d_h = 64 tokens
    # against d = 512 proxies): ragged with two sequences, 8x8 factors,
    # bidirectional add injection with 128-wide tokens
    "asym_dfine64_d512_P64_ragged_b2": (S.LayerSpec(batch=2, L=2000, d=512, n_heads=8, P=64,
                                                    d_fine=64), True, False),
    "asym_dfine64_d512_P64_8x8": (S.LayerSpec(batch=1, L=8192, d=512, n_heads=8, P=64, levels=2,
                                              k1=8, k2=8, d_fine=64), False, False),
    "asym_bidir_add_dfine128": (S.LayerSpec(batch=1, L=1024, d=256, n_heads=4, P=16,
                                            mode=S.BIDIR_1D, inject=S.INJ_ADD, d_fine=128),
                                False, False),
    # proxy interaction variants (Sec. 3.4): single-proxy MLP, identity, and
    # attention with RoPE on the proxies' queries and keys
    "mlp_causal_gated_2lvl_ragged_b2": (S.LayerSpec(batch=2, L=2000, d=128, n_heads=2, P=16,
                                                    levels=2, k1=4, k2=4, interact=S.F_MLP),
                                        True, False),
    "mlp_d1024_P64": (S.LayerSpec(batch=1, L=8192, d=1024, n_heads=16, P=64, interact=S.F_MLP),
                      False, False),
    "identity_bidir_add_b2": (S.LayerSpec(batch=2, L=1000, d=128, n_heads=2, P=16,
                                          mode=S.BIDIR_1D, inject=S.INJ_ADD,
                                          interact=S.F_IDENTITY), True, False),
    "rope_causal_gated_b2": (S.LayerSpec(batch=2, L=4000, d=128, n_heads=2, P=16, rope=1),
                             True, False),
    "rope_d1024_P64_8x8": (S.LayerSpec(batch=1, L=16384, d=1024, n_heads=16, P=64, levels=2,
                                       k1=8, k2=8, rope=1), False, False),
}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pf.build()
    pf.load()


def _stream():
    return torch.cuda.current_stream().cuda_stream


def run_gpu(spec, inp, with_h_in):
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.bfloat16)
    G = to_device(inp["G"], torch.bfloat16)
    H_in = to_device(inp["H_in"], torch.float32) if with_h_in else None
    dHo = to_device(inp["dH_out"], torch.float32)
    H_out, dH_in = lay.empty_proxy(), lay.empty_proxy()
    Xo = lay.forward(X, H_in, H_out=H_out)
    dX = lay.backward(X, G, H_in, dH_out=dHo, dH_in=dH_in)
    pf.pf_sync_check(_stream())
    f = lambda t: t.float().cpu().numpy()
    return dict(Xo=f(Xo), H=f(H_out), dX=f(dX), dH=f(dH_in),
                grads={k: f(v) for k, v in lay.grads.items()}), lay


@pytest.mark.parametrize("name", list(CASES))
def test_layer_fwd_bwd_matches_oracle(name):
    spec, with_h_in, strict = CASES[name]
    inp = S.make_layer_inputs(spec, 100 + len(name), with_h_in=with_h_in)
    got, _ = run_gpu(spec, inp, with_h_in)
    H_in = inp.get("H_in")
    Xo, H = OL.layer_fwd(spec, inp, inp["X"], H_in)
    dX, dH, grads = OL.layer_bwd(spec, inp, inp["X"], inp["G"], H_in, None, inp["dH_out"])
    # the cross injection's bf16 floor is higher (test_bf16_error_floor.py):
    # X_out up to 5e-2 max, gradients up to 2.3e-1 max and 2e-2 RMS
    cross = spec.inject == S.INJ_CROSS
    tol, max_tol = (CROSS_TOL, CROSS_MAX_TOL) if cross else (2e-2, 1e-1)
    if strict and not cross:
        assert_close("X_out", got["Xo"], Xo)
    else:
        assert_grad_close("X_out", got["Xo"], Xo)
    assert_update_close("X_out - X", inp["X"], got["Xo"], Xo, max_tol=2e-1 if cross else 1e-1)
    assert_close("H_out", got["H"], H)
    assert_grad_close("dX", got["dX"], dX, tol, max_tol)
    assert_grad_close("dH_in", got["dH"], dH, tol, max_tol)
    for k, v in grads.items():
        assert_grad_close("grad " + k, got["grads"][k], v, tol, max_tol)


@pytest.mark.parametrize("inject", [S.INJ_GATED, S.INJ_CROSS])
def test_layer_deterministic_and_causal(inject):
    """Two runs are bit-identical; perturbing token t0 leaves every output
    before the end of its block bit-identical except t0 (causal routing)."""
    spec = S.LayerSpec(batch=1, L=2000, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4,
                       inject=inject)
    inp = S.make_layer_inputs(spec, 7, with_grads=False)
    lay = ProxyLayer(spec, inp)
    X = to_device(inp["X"], torch.bfloat16)
    a = lay.forward(X, train=False).clone()
    b = lay.forward(X, train=False).clone()
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    for t0 in (0, 17, 999, 1999):
        X2 = X.clone()
        X2[0, t0] += 1.0
        c = lay.forward(X2, train=False)
        torch.cuda.synchronize()
        lim = (t0 // spec.P + 1) * spec.P
        keep = torch.ones(spec.L, dtype=torch.bool, device="cuda")
        keep[t0] = False
        keep[lim:] = False
        assert torch.equal(a[0][keep], c[0][keep]), t0
        if lim < spec.L:
            assert not torch.equal(a[0, lim:], c[0, lim:])


def test_block_routing_probe():
    """Uniform attention (W_q = W_k = 0) over one-hot-free proxies H_in[i] =
    2**i e_0 and a decompression copying channel 0: token t must receive
    mean_{j<b} 2**j with b = t // P its block; decoded to the nearest
    candidate, the block index must be exact for every token."""
    P, m, d = 16, 12, 64
    spec = S.LayerSpec(batch=2, L=P * m - 5, d=d, n_heads=1, P=P, inject=S.INJ_ADD)
    prm = S.make_layer_params(spec, 0)
    prm["W_c1"][:] = 0
    prm["b_c1"][:] = 0
    prm["W_qkv"] = np.concatenate([np.zeros((2 * d, d)), np.eye(d)]).astype(np.float32)
    prm["W_o"] = np.eye(d, dtype=np.float32)
    prm["W_d1"] = np.zeros((P * d, d), np.float32)
    prm["W_d1"][:, 0] = 1
    prm["b_d1"][:] = 0
    lay = ProxyLayer(spec, prm)
    H_in = torch.zeros(2, m, d, device="cuda")
    H_in[:, :, 0] = 2.0 ** torch.arange(m, device="cuda")
    X = torch.zeros(2, spec.L, d, dtype=torch.bfloat16, device="cuda")
    out = lay.forward(X, H_in, train=False).float().cpu().numpy()
    cand = np.array([0.0] + [np.mean(2.0 ** np.arange(b)) for b in range(1, m + 1)])
    for bb in range(2):
        for t in range(spec.L):
            row = out[bb, t]
            assert np.ptp(row) == 0.0
            assert int(np.argmin(np.abs(cand - row[0]))) == t // P, (bb, t, row[0])
