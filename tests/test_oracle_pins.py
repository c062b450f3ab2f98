"""Pins of the float64 oracle against facts fixed by the paper or by mathematics.

Each test below ties one oracle function to something other than itself: a
library routine on a special case that reduces to it, brute force on tiny
inputs, an exact invariant, an algebraic identity, or central finite
differences.  All run on the CPU (no GPU marker).
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.linalg
import scipy.special
import torch
import torch.nn.functional as F

import pf_synth as S
from oracle import layer as OL
from oracle import decode as OD

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _spec(**kw):
    base = dict(batch=1, L=12, d=8, n_heads=2, P=1, dtype=S.F32)
    base.update(kw)
    return S.LayerSpec(**base)


def _identity_params(spec, rng):
    """P=1 layer whose compression, decompression and output projection are
    identities; W_q/W_k/W_v random; gate weights zero (Pin P1)."""
    d = spec.d
    prm = S.make_layer_params(spec, 7)
    prm["W_c1"] = np.eye(d)
    prm["b_c1"] = np.zeros(d)
    prm["W_o"] = np.eye(d)
    prm["W_d1"] = np.eye(d)
    prm["b_d1"] = np.zeros(d)
    if spec.inject == S.INJ_GATED:
        prm["w_x"] = np.zeros(d)
        prm["w_dlt"] = np.zeros(d)
        prm["b_g"] = rng.uniform(-1, 1, d)
    return prm


def _sdpa(X, Wqkv, nh, causal):
    """torch SDPA (CPU, float64) on the per-head projections of X [L, d]."""
    L, d = X.shape
    dh = d // nh
    Xt = torch.from_numpy(X)
    W = torch.from_numpy(np.asarray(Wqkv, dtype=np.float64))
    q, k, v = (Xt @ W[i * d:(i + 1) * d].T for i in range(3))
    sh = lambda a: a.reshape(L, nh, dh).transpose(0, 1).unsqueeze(0)
    o = F.scaled_dot_product_attention(sh(q), sh(k), sh(v), is_causal=causal)
    return o.squeeze(0).transpose(0, 1).reshape(L, d).numpy()


# ----------------------------------------------------------------- P1
@pytest.mark.parametrize("inject", [S.INJ_GATED, S.INJ_ADD])
def test_p1_causal_reduces_to_sdpa_shifted(inject):
    """Eq. proxy-attn with P=1 and identity C, D, W_o is ordinary causal
    attention; the causal routing shifts it by one token, and the gate with
    w_x = w_dlt = 0 scales it by sigmoid(b_g) (Eq. inj-gate)."""
    rng = np.random.default_rng(0)
    spec = _spec(inject=inject)
    prm = _identity_params(spec, rng)
    X = rng.standard_normal((1, spec.L, spec.d))
    Xo, H = OL.layer_fwd(spec, prm, X)
    ref = _sdpa(X[0], prm["W_qkv"], spec.n_heads, causal=True)
    upd = Xo[0] - X[0]
    if inject == S.INJ_GATED:
        upd = upd / OL.sigmoid(prm["b_g"])
    np.testing.assert_allclose(upd[0], 0.0, atol=0)
    np.testing.assert_allclose(upd[1:], ref[:-1], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(H[0], X[0], rtol=0, atol=0)


def test_p1_bidirectional_reduces_to_sdpa():
    rng = np.random.default_rng(1)
    spec = _spec(mode=S.BIDIR_1D, inject=S.INJ_ADD)
    prm = _identity_params(spec, rng)
    X = rng.standard_normal((1, spec.L, spec.d))
    Xo, _ = OL.layer_fwd(spec, prm, X)
    ref = _sdpa(X[0], prm["W_qkv"], spec.n_heads, causal=False)
    np.testing.assert_allclose(Xo[0] - X[0], ref, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------- P2
@pytest.mark.parametrize("causal", [True, False])
def test_p2_bruteforce_masked_softmax(causal):
    """Explicit m x m score matrix with -inf entries and a full softmax."""
    rng = np.random.default_rng(2)
    spec = _spec(L=9, d=12, n_heads=3, mode=S.CAUSAL_1D if causal else S.BIDIR_1D)
    prm = S.make_layer_params(spec, 3)
    H = rng.standard_normal((spec.L, spec.d))
    Hbar, _ = OL.attention(H, prm, spec)
    d, nh = spec.d, spec.n_heads
    dh = d // nh
    W = prm["W_qkv"].astype(np.float64)
    Q, K, V = H @ W[:d].T, H @ W[d:2 * d].T, H @ W[2 * d:].T
    m = spec.L
    M = np.where(np.tril(np.ones((m, m))) > 0, 0.0, -np.inf) if causal else np.zeros((m, m))
    A = np.zeros((m, d))
    for h in range(nh):
        cs = slice(h * dh, (h + 1) * dh)
        Sm = Q[:, cs] @ K[:, cs].T / math.sqrt(dh) + M
        A[:, cs] = scipy.special.softmax(Sm, axis=1) @ V[:, cs]
    np.testing.assert_allclose(Hbar, A @ prm["W_o"].astype(np.float64).T, rtol=1e-12, atol=1e-13)


# ----------------------------------------------------------------- P3
def test_p3_mask_support_is_exactly_causal():
    """One-hot values (V_j = e_j) expose which keys each query reads: the
    support of output row i must be exactly {j <= i}."""
    m = 16
    spec = _spec(L=m, d=m, n_heads=1, mode=S.CAUSAL_1D)
    rng = np.random.default_rng(4)
    prm = {"W_qkv": np.concatenate([rng.standard_normal((m, m)) * 0.1,
                                    rng.standard_normal((m, m)) * 0.1, np.eye(m)]),
           "W_o": np.eye(m)}
    Hbar, _ = OL.attention(np.eye(m), prm, spec)
    support = Hbar != 0.0
    assert (support == (np.tril(np.ones((m, m))) > 0)).all()


def test_p3_block_routing_probe():
    """Routing probe: W_q = W_k = 0 makes every visible key equally likely, so
    Hbar_i = mean_{j<=i} H_j; H_in[i] = 2**i encodes the proxy index and
    W_d1 copies channel 0 everywhere.  Token t must then receive exactly
    mean_{j<=b-1} 2**j with b = t // P its block (0 for block 0)."""
    P, m, d = 4, 6, 4
    spec = _spec(L=P * m - 2, d=d, n_heads=1, P=P, inject=S.INJ_ADD)
    prm = S.make_layer_params(spec, 0)
    prm["W_c1"] = np.zeros_like(prm["W_c1"])
    prm["b_c1"] = np.zeros(d)
    prm["W_qkv"] = np.concatenate([np.zeros((2 * d, d)), np.eye(d)])
    prm["W_o"] = np.eye(d)
    Wd = np.zeros((P * d, d))
    Wd[:, 0] = 1.0
    prm["W_d1"] = Wd
    prm["b_d1"] = np.zeros(P * d)
    H_in = np.zeros((1, m, d))
    H_in[0, :, 0] = 2.0 ** np.arange(m)
    X = np.zeros((1, spec.L, d))
    Xo, _ = OL.layer_fwd(spec, prm, X, H_in=H_in)
    cand = np.array([0.0] + [np.mean(2.0 ** np.arange(b)) for b in range(1, m + 1)])
    for t in range(spec.L):
        got = Xo[0, t]
        assert np.ptp(got) == 0.0
        decoded = int(np.argmin(np.abs(cand - got[0])))
        assert decoded == t // P and abs(cand[decoded] - got[0]) < 1e-12, (t, got, decoded)


# ----------------------------------------------------------------- P4
@pytest.mark.parametrize("levels", [1, 2])
def test_p4_causality_perturbation(levels):
    """Perturbing X[t0] leaves X_out bit-identical at every t < (t0//P+1)*P
    except t0 itself, and does change later blocks."""
    P = 4
    spec = S.LayerSpec(batch=1, L=22, d=8, n_heads=2, P=P, levels=levels,
                       k1=2 if levels == 2 else 0, k2=2 if levels == 2 else 0, dtype=S.F32)
    inp = S.make_layer_inputs(spec, 5, with_grads=False)
    X = inp["X"].astype(np.float64)
    Xo, _ = OL.layer_fwd(spec, inp, X)
    for t0 in (0, 5, 13, 21):
        X2 = X.copy()
        X2[0, t0] += 0.75
        Xo2, _ = OL.layer_fwd(spec, inp, X2)
        lim = (t0 // P + 1) * P
        same = np.ones(spec.L, bool)
        same[t0] = False
        assert (Xo2[0, :lim][same[:lim]] == Xo[0, :lim][same[:lim]]).all()
        if lim < spec.L:
            assert np.abs(Xo2[0, lim:] - Xo[0, lim:]).max() > 1e-6


# ----------------------------------------------------------------- P5
def _loss(spec, prm, X, H_in, t, G, dHo):
    Xo, H = OL.layer_fwd(spec, prm, X, H_in, t)
    return float((Xo * G).sum() + (H * dHo).sum())


FD_SPECS = {
    "causal_gated_1lvl": S.LayerSpec(batch=2, L=30, d=8, n_heads=2, P=4, dtype=S.F32),
    "causal_gated_2lvl": S.LayerSpec(batch=1, L=32, d=8, n_heads=2, P=4, levels=2, k1=2, k2=2,
                                     dtype=S.F32),
    "bidir_add_2lvl": S.LayerSpec(batch=1, L=24, d=8, n_heads=2, P=4, levels=2, k1=2, k2=2,
                                  mode=S.BIDIR_1D, inject=S.INJ_ADD, dtype=S.F32),
    "2d_affine": S.LayerSpec(batch=2, L=64, d=8, n_heads=2, P=4, mode=S.BIDIR_2D,
                             inject=S.INJ_AFFINE, grid_h=8, grid_w=8, patch=2, dtype=S.F32),
    "causal_cross_1lvl": S.LayerSpec(batch=2, L=22, d=8, n_heads=2, P=4, inject=S.INJ_CROSS,
                                     dtype=S.F32),
    "causal_gated_2lvl_dfine4": S.LayerSpec(batch=2, L=22, d=8, n_heads=2, P=4, levels=2, k1=2,
                                            k2=2, d_fine=4, dtype=S.F32),
    "causal_gated_mlp": S.LayerSpec(batch=2, L=22, d=8, n_heads=2, P=4, interact=S.F_MLP,
                                    dtype=S.F32),
    "bidir_add_identity_2lvl": S.LayerSpec(batch=1, L=24, d=8, n_heads=2, P=4, levels=2, k1=2,
                                           k2=2, mode=S.BIDIR_1D, inject=S.INJ_ADD,
                                           interact=S.F_IDENTITY, dtype=S.F32),
    "causal_gated_rope": S.LayerSpec(batch=2, L=30, d=8, n_heads=2, P=4, rope=1, dtype=S.F32),
    "bidir_cross_2lvl": S.LayerSpec(batch=1, L=24, d=8, n_heads=2, P=4, levels=2, k1=2, k2=2,
                                    mode=S.BIDIR_1D, inject=S.INJ_CROSS, dtype=S.F32),
}


@pytest.mark.parametrize("name", sorted(FD_SPECS))
def test_p5_finite_differences(name):
    spec = FD_SPECS[name]
    inp = S.make_layer_inputs(spec, 11, with_h_in=True)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    X, H_in, G, dHo = prm["X"], prm["H_in"], prm["G"], prm["dH_out"]
    t = prm.get("t")
    dX, dH_in, grads = OL.layer_bwd(spec, prm, X, G, H_in, t, dHo)
    rng = np.random.default_rng(12)
    eps = 1e-6
    targets = dict(grads)
    targets["X"] = dX
    targets["H_in"] = dH_in
    for key, an in targets.items():
        base = prm[key]
        flat = base.reshape(-1)
        idx = rng.choice(flat.size, size=min(12, flat.size), replace=False)
        for j in idx:
            old = flat[j]
            flat[j] = old + eps
            lp = _loss(spec, prm, X, H_in, t, G, dHo)
            flat[j] = old - eps
            lm = _loss(spec, prm, X, H_in, t, G, dHo)
            flat[j] = old
            fd = (lp - lm) / (2 * eps)
            a = an.reshape(-1)[j]
            assert abs(fd - a) <= 1e-6 * max(1.0, abs(a)), (key, j, fd, a)


# --------------------------------------------------- cross-attention injection
@pytest.mark.parametrize("causal", [True, False])
def test_cross_injection_equals_masked_sdpa(causal):
    """Gated Eq. inj-cross against torch SDPA with an explicit boolean mask
    (token t of block i sees proxies j < i when causal, all otherwise),
    projections and gate recomputed here with torch: X_out - X must equal
    (sigmoid(X W_a^T + b_a) * A) W_ox^T, and a token that sees no proxy gets
    exactly nothing."""
    P, L, d, nh = 4, 23, 8, 2
    spec = S.LayerSpec(batch=1, L=L, d=d, n_heads=nh, P=P, inject=S.INJ_CROSS, dtype=S.F32,
                       mode=S.CAUSAL_1D if causal else S.BIDIR_1D)
    prm = {k: v.astype(np.float64) for k, v in S.make_layer_params(spec, 41).items()}
    rng = np.random.default_rng(42)
    X = rng.standard_normal((L, d))
    Hbar = rng.standard_normal((spec.m, d))
    Xo, _ = OL.cross_inject(X, Hbar, prm, spec)
    T = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    Xt, Ht = T(X), T(Hbar)
    Wqa, Wkv = T(prm["W_qa"]), T(prm["W_kvx"])
    q, k, v = Xt @ Wqa[:d].T, Ht @ Wkv[:d].T, Ht @ Wkv[d:].T
    alpha = torch.sigmoid(Xt @ Wqa[d:].T + T(prm["b_a"]))
    vis = torch.ones(L, spec.m, dtype=torch.bool)
    if causal:
        vis = torch.arange(spec.m)[None, :] < (torch.arange(L) // P)[:, None]
    sh = lambda a: a.reshape(a.shape[0], nh, d // nh).transpose(0, 1)
    rows = vis.any(1)
    o = F.scaled_dot_product_attention(sh(q[rows]), sh(k), sh(v), attn_mask=vis[rows])
    A = torch.zeros(L, d, dtype=torch.float64)
    A[rows] = o.transpose(0, 1).reshape(-1, d)
    ref = X + ((A.reshape(L, nh, -1) * alpha[:, :, None]).reshape(L, d) @ T(prm["W_ox"]).T).numpy()
    np.testing.assert_allclose(Xo, ref, rtol=1e-12, atol=1e-12)
    if causal:
        assert (Xo[:P] == X[:P]).all()


def test_cross_injection_routing_probe():
    """Uniform attention (W_q = 0) over proxies Hbar_j = 2^j e_0 with identity
    W_v and W_ox and a zero gate map (alpha = 1/2): token t must receive
    mean_{j < t//P} 2^j / 2 (to rounding) in every channel, which decodes the
    set of proxies it read."""
    P, m, d = 4, 6, 4
    spec = S.LayerSpec(batch=1, L=P * m - 1, d=d, n_heads=1, P=P, inject=S.INJ_CROSS,
                       dtype=S.F32)
    prm = {"W_qa": np.zeros((d + 1, d)), "b_a": np.zeros(1),
           "W_kvx": np.concatenate([np.eye(d), np.eye(d)]), "W_ox": np.zeros((d, d))}
    prm["W_ox"][:, 0] = 1.0
    Hbar = np.zeros((m, d))
    Hbar[:, 0] = 2.0 ** np.arange(m)
    X = np.zeros((spec.L, d))
    Xo, _ = OL.cross_inject(X, Hbar, prm, spec)
    cand = np.array([0.0] + [np.mean(2.0 ** np.arange(i)) / 2 for i in range(1, m)])
    for t in range(spec.L):
        assert np.ptp(Xo[t]) == 0.0
        i = int(np.argmin(np.abs(cand - Xo[t, 0])))
        assert i == t // P and abs(Xo[t, 0] - cand[i]) < 1e-12, (t, Xo[t], i)


@pytest.mark.parametrize("mode", [S.CAUSAL_1D, S.BIDIR_1D])
def test_cross_injection_causality(mode):
    """Causal: perturbing X[t0] leaves X_out bit-identical before the end of
    t0's block except at t0 (its own query), and changes later blocks.
    Bidirectional: later blocks' proxies reach earlier tokens."""
    P = 4
    spec = S.LayerSpec(batch=1, L=22, d=8, n_heads=2, P=P, mode=mode, inject=S.INJ_CROSS,
                       dtype=S.F32)
    inp = S.make_layer_inputs(spec, 43, with_grads=False)
    X = inp["X"].astype(np.float64)
    Xo, _ = OL.layer_fwd(spec, inp, X)
    for t0 in (1, 9, 21):
        X2 = X.copy()
        X2[0, t0] += 0.75
        Xo2, _ = OL.layer_fwd(spec, inp, X2)
        lim = (t0 // P + 1) * P
        same = np.ones(spec.L, bool)
        same[t0] = False
        if mode == S.CAUSAL_1D:
            assert (Xo2[0, :lim][same[:lim]] == Xo[0, :lim][same[:lim]]).all()
            if lim < spec.L:
                assert np.abs(Xo2[0, lim:] - Xo[0, lim:]).max() > 1e-6
        else:
            assert np.abs(Xo2[0, :t0 // P * P] - Xo[0, :t0 // P * P]).max(initial=1.0) > 1e-6


# ------------------------------------------------------ asymmetric widths
@pytest.mark.parametrize("inject,levels", [(S.INJ_GATED, 2), (S.INJ_ADD, 1)])
def test_asymmetric_widths_embed_in_a_symmetric_layer(inject, levels):
    """A layer with d_fine = 4-wide tokens and d = 8-wide proxies equals the
    symmetric d = 8 layer run on the tokens zero-padded to 8 channels, when
    that layer's compression reads the real channels with the same weights
    (its weights on the padding channels are arbitrary: they multiply zeros)
    and its decompression writes zero into the padding channels.  The padded
    channels of X_out must stay exactly zero."""
    kw = dict(batch=2, L=22, d=8, n_heads=2, P=4, levels=levels, inject=inject, dtype=S.F32,
              k1=2 if levels == 2 else 0, k2=2 if levels == 2 else 0)
    sa, ss = S.LayerSpec(d_fine=4, **kw), S.LayerSpec(**kw)
    pa = {k: v.astype(np.float64) for k, v in S.make_layer_params(sa, 51).items()}
    ps = {k: v.astype(np.float64) for k, v in S.make_layer_params(ss, 52).items()}
    k1, df, d = sa.k1, 4, 8
    for k in ("b_c1", "W_c2", "b_c2", "W_qkv", "W_o", "W_d2", "b_d2"):
        if k in pa:
            ps[k] = pa[k]
    for t in range(k1):  # token slot t of a k1-group: channels [t*d, t*d + df)
        ps["W_c1"][:, t * d:t * d + df] = pa["W_c1"][:, t * df:(t + 1) * df]
        ps["W_d1"][t * d:(t + 1) * d] = 0.0
        ps["W_d1"][t * d:t * d + df] = pa["W_d1"][t * df:(t + 1) * df]
        ps["b_d1"][t * d:(t + 1) * d] = 0.0
        ps["b_d1"][t * d:t * d + df] = pa["b_d1"][t * df:(t + 1) * df]
    if inject == S.INJ_GATED:
        for k in ("w_x", "w_dlt", "b_g"):
            ps[k][:df] = pa[k]
    rng = np.random.default_rng(53)
    Xa = rng.standard_normal((2, sa.L, df))
    Xs = np.concatenate([Xa, np.zeros((2, sa.L, d - df))], axis=2)
    H_in = rng.standard_normal((2, sa.m, d))
    oa, ha = OL.layer_fwd(sa, pa, Xa, H_in)
    os_, hs = OL.layer_fwd(ss, ps, Xs, H_in)
    np.testing.assert_allclose(oa, os_[..., :df], rtol=1e-12, atol=1e-12)
    assert (os_[..., df:] == 0.0).all()
    np.testing.assert_allclose(ha, hs, rtol=1e-12, atol=1e-12)


# ------------------------------------------------- proxy interaction variants
def test_identity_interaction_closed_form():
    """F = identity (Hbar = H) with P = 1 and identity compression and
    decompression: each token receives the previous token (causal routing),
    the first nothing -- X_out[t] = X[t] + X[t-1] exactly."""
    spec = _spec(inject=S.INJ_ADD, interact=S.F_IDENTITY)
    d = spec.d
    prm = {"W_c1": np.eye(d), "b_c1": np.zeros(d), "W_d1": np.eye(d), "b_d1": np.zeros(d)}
    X = np.random.default_rng(61).standard_normal((1, spec.L, d))
    Xo, H = OL.layer_fwd(spec, prm, X)
    np.testing.assert_array_equal(Xo[0, 0], X[0, 0])
    np.testing.assert_array_equal(Xo[0, 1:], X[0, 1:] + X[0, :-1])
    np.testing.assert_array_equal(H[0], X[0])


def test_mlp_interaction_equals_torch():
    """The single-proxy MLP is torch's linear -> SiLU -> linear on every row."""
    spec = S.LayerSpec(batch=1, L=40, d=8, n_heads=2, P=4, interact=S.F_MLP, dtype=S.F32)
    prm = {k: v.astype(np.float64) for k, v in S.make_layer_params(spec, 62).items()}
    H = np.random.default_rng(63).standard_normal((spec.m, spec.d))
    got, _ = OL.interact(H, prm, spec)
    T = lambda a: torch.from_numpy(np.asarray(a, np.float64))
    ref = F.linear(F.silu(F.linear(T(H), T(prm["W_m1"]), T(prm["b_m1"]))), T(prm["W_m2"]),
                   T(prm["b_m2"]))
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_rope_rotation_properties():
    """RoPE on the proxies: position 0 is the identity; position 1 turns pair
    j of a head by base^(-2j/dh) radians; the inverse is the transpose; and a
    rotated query-key dot product depends only on the distance of the two
    positions (shifting both leaves it unchanged)."""
    nh, dh, m = 2, 8, 12
    d = nh * dh
    rng = np.random.default_rng(64)
    Z = rng.standard_normal((m, d))
    R = OL.rope(Z, nh)
    np.testing.assert_array_equal(R[0], Z[0])
    e = np.zeros((2, d))
    e[1, 2] = 1.0  # head 0, pair j = 1, first element, at position 1
    r = OL.rope(e, nh)[1]
    a = OL.ROPE_BASE ** (-2.0 / dh)
    np.testing.assert_allclose(r[2:4], [math.cos(a), math.sin(a)], rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(OL.rope(R, nh, inverse=True), Z, rtol=1e-12, atol=1e-12)
    q, k = rng.standard_normal(d), rng.standard_normal(d)
    def dot_at(i, j):
        Q = np.zeros((m, d)); K = np.zeros((m, d))
        Q[i], K[j] = q, k
        return float(OL.rope(Q, nh)[i] @ OL.rope(K, nh)[j])
    for i, j, s in ((5, 2, 3), (7, 7, 4), (1, 9, 2)):
        assert abs(dot_at(i, j) - dot_at(i + s, j + s)) < 1e-12


# ----------------------------------------------------------------- P6
def test_p6_factorised_equals_single_level():
    """Eq. factor-cascade with no nonlinearity is one linear map:
    W_eq = W_c2 blockdiag_k2(W_c1), b_eq = W_c2 tile(b_c1) + b_c2; the
    decompression side likewise (Eq. factor-dec)."""
    k1, k2, d = 2, 3, 4
    spec2 = S.LayerSpec(batch=2, L=30, d=d, n_heads=2, P=k1 * k2, levels=2, k1=k1, k2=k2,
                        dtype=S.F32)
    spec1 = S.LayerSpec(batch=2, L=30, d=d, n_heads=2, P=k1 * k2, dtype=S.F32)
    inp = S.make_layer_inputs(spec2, 21, with_h_in=True, with_grads=False)
    p2 = {k: v.astype(np.float64) for k, v in inp.items()}
    p1 = dict(p2)
    bd_c = scipy.linalg.block_diag(*[p2["W_c1"]] * k2)
    p1["W_c1"] = p2["W_c2"] @ bd_c
    p1["b_c1"] = p2["W_c2"] @ np.tile(p2["b_c1"], k2) + p2["b_c2"]
    bd_d = scipy.linalg.block_diag(*[p2["W_d1"]] * k2)
    p1["W_d1"] = bd_d @ p2["W_d2"]
    p1["b_d1"] = bd_d @ p2["b_d2"] + np.tile(p2["b_d1"], k2)
    for k in ("W_c2", "b_c2", "W_d2", "b_d2"):
        del p1[k]
    a = OL.layer_fwd(spec2, p2, p2["X"], p2["H_in"])
    b = OL.layer_fwd(spec1, p1, p2["X"], p2["H_in"])
    np.testing.assert_allclose(a[0], b[0], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(a[1], b[1], rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------- P7
def test_p7_2d_compression_is_conv_and_decompression_is_conv_transpose():
    """Sec. 3.2/3.5: 2D patch compression is conv2d with kernel = stride = p,
    and the affine decompression is the matching conv_transpose2d."""
    spec = S.LayerSpec(batch=1, L=36, d=4, n_heads=2, P=4, mode=S.BIDIR_2D,
                       inject=S.INJ_AFFINE, grid_h=6, grid_w=6, patch=2, dtype=S.F32)
    inp = S.make_layer_inputs(spec, 31, with_grads=False)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    p, d = spec.patch, spec.d
    X = prm["X"][0]
    C, _ = OL.compress(OL.partition(X, spec), prm, spec)
    w = torch.from_numpy(prm["W_c1"].reshape(d, p, p, d).transpose(0, 3, 1, 2).copy())
    img = torch.from_numpy(X.reshape(6, 6, d).transpose(2, 0, 1).copy()).unsqueeze(0)
    conv = F.conv2d(img, w, torch.from_numpy(prm["b_c1"]), stride=p)[0]
    np.testing.assert_allclose(C, conv.permute(1, 2, 0).reshape(-1, d).numpy(), rtol=1e-12,
                               atol=1e-12)
    Hbar = np.random.default_rng(3).standard_normal(C.shape)
    D, _ = OL.decompress(Hbar, prm, spec)
    Dt = OL.unpartition(D, spec, spec.L)                        # [L, 2d]
    wt = torch.from_numpy(prm["W_d1"].reshape(p, p, 2 * d, d).transpose(3, 2, 0, 1).copy())
    hb = torch.from_numpy(Hbar.reshape(3, 3, d).transpose(2, 0, 1).copy()).unsqueeze(0)
    up = F.conv_transpose2d(hb, wt, stride=p)[0]                # [2d, 6, 6]
    bias = prm["b_d1"].reshape(p, p, 2 * d)
    ref = up.permute(1, 2, 0).numpy() + np.tile(bias, (3, 3, 1))
    np.testing.assert_allclose(Dt, ref.reshape(spec.L, 2 * d), rtol=1e-12, atol=1e-12)


def test_norms_match_torch():
    x = np.random.default_rng(8).standard_normal((5, 16)) * 3 + 1
    n, _, _ = OL.layernorm(x)
    ref = F.layer_norm(torch.from_numpy(x), (16,), eps=OL.LN_EPS).numpy()
    np.testing.assert_allclose(n, ref, rtol=1e-12, atol=1e-12)
    w = np.random.default_rng(9).uniform(0.5, 1.5, 16)
    r = OD.rmsnorm(x[0], w)
    ref = F.rms_norm(torch.from_numpy(x[:1]), (16,), torch.from_numpy(w), eps=OD.RMS_EPS)
    np.testing.assert_allclose(r, ref.numpy()[0], rtol=1e-12, atol=1e-12)


def test_affine_injection_with_constant_modulation():
    """Eq. inj-affine with W_d1 = 0: s and t are the per-channel biases, so
    X_out = (1 + s) LayerNorm(X) + t, LayerNorm taken from torch."""
    spec = FD_SPECS["2d_affine"]
    inp = S.make_layer_inputs(spec, 13, with_grads=False)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    prm["W_d1"] = np.zeros_like(prm["W_d1"])
    d, P = spec.d, spec.P
    s0, t0 = np.random.default_rng(1).standard_normal((2, d))
    prm["b_d1"] = np.tile(np.concatenate([s0, t0]), P)
    Xo, _ = OL.layer_fwd(spec, prm, prm["X"], t=prm["t"])
    ln = F.layer_norm(torch.from_numpy(prm["X"]), (d,), eps=OL.LN_EPS).numpy()
    np.testing.assert_allclose(Xo, (1 + s0) * ln + t0, rtol=1e-12, atol=1e-12)


def test_gate_limits_reduce_to_add_and_identity():
    """sigmoid(g) -> 1 turns Eq. inj-gate into Eq. inj-add; -> 0 leaves X;
    a steep w_x makes the gate the indicator X > 0."""
    spec = S.LayerSpec(batch=1, L=20, d=8, n_heads=2, P=4, dtype=S.F32)
    inp = S.make_layer_inputs(spec, 17, with_grads=False)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    X = prm["X"]
    add = OL.layer_fwd(S.LayerSpec(batch=1, L=20, d=8, n_heads=2, P=4, inject=S.INJ_ADD,
                                   dtype=S.F32), prm, X)[0]
    for bg, want in ((60.0, add), (-60.0, X)):
        p = dict(prm, w_x=np.zeros(8), w_dlt=np.zeros(8), b_g=np.full(8, bg))
        np.testing.assert_allclose(OL.layer_fwd(spec, p, X)[0], want, rtol=1e-13, atol=1e-13)
    p = dict(prm, w_x=np.full(8, 1e6), w_dlt=np.zeros(8), b_g=np.zeros(8))
    step = np.where(X > 0, add - X, 0.0) + X
    np.testing.assert_allclose(OL.layer_fwd(spec, p, X)[0], step, rtol=1e-13, atol=1e-13)


# ----------------------------------------------------------------- P8
def _dec_setup(n_proxy, n_open, levels=1):
    spec = S.DecodeSpec(batch=3, d=16, n_heads=2, P=4, levels=levels,
                        k1=2 if levels == 2 else 0, k2=2 if levels == 2 else 0, capacity=6)
    prm = S.make_decode_params(spec, 41)
    st = S.make_decode_state(spec, 42, n_proxy, n_open)
    return spec, prm, st


def test_p8_decode_attentions_are_sdpa():
    """Eq. llm-cross: A_x is causal SDPA of the new token over the open block,
    A_h plain SDPA over the cached proxies; two separate softmaxes."""
    spec, prm, st = _dec_setup([3, 0, 6], [2, 0, 3])
    y, new, parts = OD.decode_step(spec, prm, st, return_parts=True)
    d, nh = spec.d, spec.n_heads
    dh = d // nh
    for b in range(3):
        q = torch.from_numpy(parts[b]["q"]).reshape(1, nh, 1, dh)
        no, npx = st["n_open"][b], st["n_proxy"][b]
        sh = lambda a: torch.from_numpy(np.asarray(a, np.float64)).reshape(-1, nh, dh).transpose(0, 1).unsqueeze(0)
        ax = F.scaled_dot_product_attention(q, sh(new["K_open"][b, :no + 1]),
                                            sh(new["V_open"][b, :no + 1]))
        np.testing.assert_allclose(parts[b]["Ax"], ax.reshape(d).numpy(), rtol=1e-12, atol=1e-12)
        if npx:
            ah = F.scaled_dot_product_attention(q, sh(st["K_proxy"][b, :npx]),
                                                sh(st["V_proxy"][b, :npx]))
            np.testing.assert_allclose(parts[b]["Ah"], ah.reshape(d).numpy(), rtol=1e-12,
                                       atol=1e-12)
        else:
            assert (parts[b]["Ah"] == 0).all()
        np.testing.assert_allclose(new["K_open"][b, no], parts[b]["k"], rtol=0, atol=0)
    assert (new["n_open"] == st["n_open"] + 1).all()


def test_p8_alpha_limits():
    """alpha -> 0 removes the proxy read: y = x + W_o A_x; alpha -> 1 adds A_h."""
    spec, prm, st = _dec_setup([3, 2, 6], [2, 0, 3])
    for lim, coef in ((-60.0, 0.0), (60.0, 1.0)):
        p = dict(prm, b_a2=np.full(spec.n_heads, lim))
        y, _, parts = OD.decode_step(spec, p, st, return_parts=True)
        for b in range(3):
            A = parts[b]["Ax"] + coef * parts[b]["Ah"]
            ref = st["x"][b] + prm["W_o"].astype(np.float64) @ A
            np.testing.assert_allclose(y[b], ref, rtol=1e-13, atol=1e-13)
    # per-head gate: head 0 reads the proxies, head 1 does not
    p = dict(prm, b_a2=np.array([60.0, -60.0]))
    y, _, parts = OD.decode_step(spec, p, st, return_parts=True)
    dh = spec.d // spec.n_heads
    for b in range(3):
        A = parts[b]["Ax"].copy()
        A[:dh] += parts[b]["Ah"][:dh]
        ref = st["x"][b] + prm["W_o"].astype(np.float64) @ A
        np.testing.assert_allclose(y[b], ref, rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("levels", [1, 2])
@pytest.mark.parametrize("with_h", [False, True])
def test_prefill_equals_appends_and_decode_writes(levels, with_h):
    """Bulk prefill of a history of m P + r tokens equals the streaming path
    it replaces (Sec. 3.8): m times (P decode steps filling the open block,
    then an append), then r decode steps -- compared on every cached proxy
    row, the open block's features, keys and values, and the counters."""
    spec, prm, st = _dec_setup([0, 0, 0], [0, 0, 0], levels)
    rng = np.random.default_rng(11)
    m, r = 2, 3  # r < P
    X = rng.standard_normal((3, m * spec.P + r, spec.d))
    # H_in is a layer's proxy stream: one row per block, the partial one included
    H_in = rng.standard_normal((3, m + 1, spec.d)) if with_h else None
    for i in range(m):
        for j in range(spec.P):
            st = dict(st, x=X[:, i * spec.P + j])
            _, st = OD.decode_step(spec, prm, st)
        st = OD.kv_append(spec, prm, st, None if H_in is None else H_in[:, i])
    for j in range(r):
        st = dict(st, x=X[:, m * spec.P + j])
        _, st = OD.decode_step(spec, prm, st)
    pre = OD.kv_prefill(spec, prm, X, H_in)
    assert (pre["n_proxy"] == st["n_proxy"]).all() and (pre["n_open"] == st["n_open"]).all()
    for k in ("K_proxy", "V_proxy"):
        np.testing.assert_allclose(pre[k][:, :m], st[k][:, :m], rtol=1e-12, atol=1e-12)
    for k in ("X_open", "K_open", "V_open"):
        np.testing.assert_allclose(pre[k][:, :r], st[k][:, :r], rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("levels", [1, 2])
def test_p8_streaming_append_equals_layer_compression(levels):
    """P decode steps fill the open block; the append then caches the same
    proxy the layer's compression (Eq. compress-linear, Eq. proxy-res) makes
    of that block, projected by W_kh / W_vh."""
    spec, prm, st = _dec_setup([1, 0, 2], [0, 0, 0], levels)
    rng = np.random.default_rng(5)
    toks = rng.standard_normal((spec.P, 3, spec.d))
    for j in range(spec.P):
        st = dict(st, x=toks[j])
        _, st = OD.decode_step(spec, prm, st)
    assert (st["n_open"] == spec.P).all()
    H_in = rng.standard_normal((3, spec.d))
    new = OD.kv_append(spec, prm, st, H_in)
    lspec = S.LayerSpec(batch=1, L=spec.P, d=spec.d, n_heads=spec.n_heads, P=spec.P,
                        levels=levels, k1=spec.k1, k2=spec.k2, dtype=S.F32)
    lprm = {k: v for k, v in prm.items() if k in ("W_c1", "b_c1", "W_c2", "b_c2")}
    W = prm["W_kvh"].astype(np.float64)
    for b in range(3):
        C, _ = OL.compress(OL.partition(toks[:, b], lspec), lprm, lspec)
        Hb = C[0] + H_in[b]
        npx = st["n_proxy"][b]
        np.testing.assert_allclose(new["K_proxy"][b, npx], W[:spec.d] @ Hb, rtol=1e-12,
                                   atol=1e-12)
        np.testing.assert_allclose(new["V_proxy"][b, npx], W[spec.d:] @ Hb, rtol=1e-12,
                                   atol=1e-12)
    assert (new["n_open"] == 0).all() and (new["n_proxy"] == st["n_proxy"] + 1).all()


# ----------------------------------------------------------------- P9
def test_p9_null_h_in_equals_zero_h_in():
    """Eq. proxy-res: without an incoming proxy state, H^(l-1) = 0."""
    spec = S.LayerSpec(batch=2, L=16, d=8, n_heads=2, P=4, dtype=S.F32)
    inp = S.make_layer_inputs(spec, 3, with_grads=False)
    a = OL.layer_fwd(spec, inp, inp["X"])
    b = OL.layer_fwd(spec, inp, inp["X"], H_in=np.zeros((2, spec.m, 8)))
    assert (a[0] == b[0]).all() and (a[1] == b[1]).all()


# ----------------------------------------------------------- golden: Sec. 4
def test_golden_complexity_ratios():
    """Sec. 4 prints, for P=64, a 4096x cheaper proxy attention and a 64x
    smaller history cache.  Count the oracle's score evaluations (the visible
    (query, key) pairs of the mask it applies) for bidirectional attention
    over L tokens vs over L/P proxies, and its cache rows after streaming L_h
    tokens."""
    with open(os.path.join(GOLDEN, "complexity_p64.json")) as f:
        g = json.load(f)
    P = g["P"]
    calls = []
    orig = OL.proxy_mask

    def counting(m, spec):
        vis = orig(m, spec)
        calls.append(int(vis.sum()))
        return vis

    OL.proxy_mask = counting
    try:
        L, d = 2 * P, 1
        full = S.LayerSpec(batch=1, L=L, d=d, n_heads=1, P=1, mode=S.BIDIR_1D, inject=S.INJ_ADD,
                           dtype=S.F32)
        prox = S.LayerSpec(batch=1, L=L, d=d, n_heads=1, P=P, mode=S.BIDIR_1D, inject=S.INJ_ADD,
                           dtype=S.F32)
        for sp in (full, prox):
            calls.clear()
            OL.attention(np.ones((sp.m, d)), {"W_qkv": np.ones((3, 1)), "W_o": np.ones((1, 1))}, sp)
            sp_count = sum(calls)
            if sp is full:
                n_full = sp_count
            else:
                n_prox = sp_count
    finally:
        OL.proxy_mask = orig
    assert n_full // n_prox == g["attention_speedup"]
    spec = S.DecodeSpec(batch=1, d=4, n_heads=1, P=P, capacity=4)
    prm = S.make_decode_params(spec, 1)
    st = S.make_decode_state(spec, 2, [0], [0])
    for blk in range(2):
        for j in range(P):
            st = dict(st, x=np.full((1, 4), 0.1 * j))
            _, st = OD.decode_step(spec, prm, st)
        st = OD.kv_append(spec, prm, st)
    assert (2 * P) // int(st["n_proxy"][0]) == g["kv_cache_compression"]


# ------------------------------------- temporal-distance ratios (Sec. 3.6)
_SEG_KEYS = ("W_c1", "b_c1", "W_c2", "b_c2", "W_d1", "b_d1", "W_d2", "b_d2")


def _split(prm):
    seg = {k: v for k, v in prm.items() if k in _SEG_KEYS}
    shared = {k: v for k, v in prm.items() if k not in _SEG_KEYS and k.startswith(("W_", "w_", "b_"))}
    return seg, shared


@pytest.mark.parametrize("levels", [1, 2])
def test_segments_one_segment_is_the_layer(levels):
    """A single segment is the ordinary causal layer, ragged tail included."""
    kw = dict(k1=2, k2=2) if levels == 2 else {}
    spec = S.LayerSpec(batch=1, L=22, d=8, n_heads=2, P=4, levels=levels, dtype=S.F32, **kw)
    inp = S.make_layer_inputs(spec, 71, with_grads=False)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    seg, shared = _split(prm)
    segs = [(22, 4, 2, 2)] if levels == 2 else [(22, 4)]
    Xo, _ = OL.layer_fwd_segments(spec, segs, [seg], shared, prm["X"][0])
    ref, _ = OL.layer_fwd(spec, prm, prm["X"])
    np.testing.assert_allclose(Xo, ref[0], rtol=1e-12, atol=1e-12)


def test_segments_equal_ratio_split_is_the_layer():
    """Two segments with the same block size and the same weights are the
    ordinary layer over their concatenation: the routing across the segment
    boundary (the first block of segment 2 receives the last proxy of
    segment 1) and the shared attention must line up exactly."""
    spec = S.LayerSpec(batch=1, L=30, d=8, n_heads=2, P=4, dtype=S.F32)
    inp = S.make_layer_inputs(spec, 72, with_grads=False)
    prm = {k: v.astype(np.float64) for k, v in inp.items()}
    seg, shared = _split(prm)
    Xo, _ = OL.layer_fwd_segments(spec, [(12, 4), (18, 4)], [seg, seg], shared, prm["X"][0])
    ref, _ = OL.layer_fwd(spec, prm, prm["X"])
    np.testing.assert_allclose(Xo, ref[0], rtol=1e-12, atol=1e-12)


def _seg_case():
    """Coarse blocks (P = 8) for the distant 16 tokens, fine (P = 4) for the
    recent 14."""
    specs = [S.LayerSpec(batch=1, L=16, d=8, n_heads=2, P=8, dtype=S.F32),
             S.LayerSpec(batch=1, L=14, d=8, n_heads=2, P=4, dtype=S.F32)]
    seg_prm, shared = [], None
    for i, sp in enumerate(specs):
        p = {k: v.astype(np.float64) for k, v in S.make_layer_params(sp, 73 + i).items()}
        sgp, sh = _split(p)
        seg_prm.append(sgp)
        shared = shared or sh
    rng = np.random.default_rng(75)
    return specs[1], [(16, 8), (14, 4)], seg_prm, shared, rng.standard_normal((30, 8)), \
        rng.standard_normal((30, 8))


def test_segments_causality():
    """Coarse-then-fine blocks keep causality: perturbing X[t0] leaves every
    output before the end of t0's block bit-identical except t0 itself."""
    spec, segs, seg_prm, shared, X, _ = _seg_case()
    Xo, _ = OL.layer_fwd_segments(spec, segs, seg_prm, shared, X)
    ends = [8, 16, 20, 24, 28, 30]  # block ends: two P = 8 blocks, then P = 4 blocks
    for t0 in (3, 12, 17, 29):
        X2 = X.copy()
        X2[t0] += 0.5
        Xo2, _ = OL.layer_fwd_segments(spec, segs, seg_prm, shared, X2)
        lim = next(e for e in ends if e > t0)
        same = np.ones(30, bool)
        same[t0] = False
        assert (Xo2[:lim][same[:lim]] == Xo[:lim][same[:lim]]).all(), t0
        if lim < 30:
            assert np.abs(Xo2[lim:] - Xo[lim:]).max() > 1e-6


def test_segments_finite_differences():
    spec, segs, seg_prm, shared, X, G = _seg_case()
    dX, sgr, gr = OL.layer_bwd_segments(spec, segs, seg_prm, shared, X, G)
    loss = lambda: float((OL.layer_fwd_segments(spec, segs, seg_prm, shared, X)[0] * G).sum())
    rng = np.random.default_rng(76)
    eps = 1e-6
    targets = [("X", X, dX)] + [(f"shared {k}", shared[k], gr[k]) for k in shared] + \
        [(f"seg{i} {k}", seg_prm[i][k], sgr[i][k]) for i in range(2) for k in seg_prm[i]]
    for name, base, an in targets:
        flat = base.reshape(-1)
        for j in rng.choice(flat.size, size=min(8, flat.size), replace=False):
            old = flat[j]
            flat[j] = old + eps
            lp = loss()
            flat[j] = old - eps
            lm = loss()
            flat[j] = old
            fd = (lp - lm) / (2 * eps)
            a = an.reshape(-1)[j]
            assert abs(fd - a) <= 1e-6 * max(1.0, abs(a)), (name, j, fd, a)
