"""Error floor of a bf16 implementation of the layer, and the tolerance it sets.

The float64 oracle's equations are evaluated again with their intermediates
rounded to bf16 at the points where the CUDA library stores bf16 tensors (Y, H
before the Q/K/V projection, Q/K/V, the probabilities fed to P.V, the attention
output, Hbar, Z, the saved D, X_out, and on the backward dD, dZ, dHbar, dA,
dS, dQKV, dH, dY, dX).  Any correct bf16 path makes errors of this size.  The
test fixes two facts the parity tolerances rely on:
  * max|err| / RMS exceeds 2e-2 for several gradients, so the max-abs bar can
    only apply to the forward outputs (X_out stays below it);
  * RMS(err) / RMS is below 1e-2 for every output, so an RMS-normalised bar of
    2e-2 (with a 1e-1 max bound) has margin for a correct kernel and still
    fails on a wrong block, sign or index (those move a whole tensor).
CPU only; it does not touch the CUDA library.
"""
import math

import numpy as np

import pf_synth as S
from oracle import layer as OL


def rb(a):
    return S.round_bf16(np.asarray(a, np.float32)).astype(np.float64)

def run(spec, p, X, G, dHo, F, H_in=None):
    f = lambda n, a: rb(a) if n in F else a
    L, d = X.shape; m = spec.m; nh = spec.n_heads; dh = d // nh; k1, k2, P = spec.k1, spec.k2, spec.P
    Xb = OL.partition(X, spec)
    groups = Xb.reshape(m, k2, k1*d)
    Y = groups @ p["W_c1"].T + p["b_c1"]
    if spec.levels == 2:
        Yr = f("Y", Y)
        H = Yr.reshape(m, k2*d) @ p["W_c2"].T + p["b_c2"]
    else:
        H = Y.reshape(m, d); Yr = None
    if H_in is not None:
        H = H + H_in
    Hq = f("H", H)
    W = p["W_qkv"]
    Q, K, V = f("QK", Hq @ W[:d].T), f("QK", Hq @ W[d:2*d].T), f("V", Hq @ W[2*d:].T)
    A = np.zeros((m, d)); Ps = []
    causal = spec.mode == 0
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh)
        Sm = Q[:, cs] @ K[:, cs].T / math.sqrt(dh)
        if causal: Sm = np.where(np.tril(np.ones((m, m))) > 0, Sm, -np.inf)
        Pm = np.exp(Sm - Sm.max(1, keepdims=True)); Pm /= Pm.sum(1, keepdims=True)
        Ps.append(Pm)
        A[:, cs] = f("P", Pm) @ V[:, cs]
    A = f("A", A)
    Hbar = f("Hbar", A @ p["W_o"].T)
    if spec.levels == 2:
        Z = f("Z", Hbar @ p["W_d2"].T + p["b_d2"]); rows = Z.reshape(m, k2, d)
    else:
        Z = None; rows = Hbar.reshape(m, 1, d)
    out = rows @ p["W_d1"].T + p["b_d1"]
    D = out.reshape(m, P, d)
    Ds = f("D", D)  # saved copy used in bwd
    Dr = np.zeros_like(D); Dr[1:] = D[:-1]; Dt = OL.unpartition(Dr, spec, L)
    Dsr = np.zeros_like(D); Dsr[1:] = Ds[:-1]; Dst = OL.unpartition(Dsr, spec, L)
    g = p["w_x"]*X + p["w_dlt"]*Dt + p["b_g"]; s = OL.sigmoid(g)
    Xo = f("Xo", X + s*Dt)
    # backward
    gs = p["w_x"]*X + p["w_dlt"]*Dst + p["b_g"]; s2 = OL.sigmoid(gs)
    ds = G*Dst*s2*(1-s2)
    dXd = G + ds*p["w_x"]
    dDt = f("dD", G*s2 + ds*p["w_dlt"])
    gr = {}
    gr["w_x"] = (ds*X).sum(0); gr["w_dlt"] = (ds*Dst).sum(0); gr["b_g"] = ds.sum(0)
    pad = np.zeros((m*P, d)); pad[:L] = dDt; dDr = pad.reshape(m, P, d)
    dD = np.zeros_like(dDr); dD[:-1] = dDr[1:]
    dout = dD.reshape(m, k2, k1*d)
    gr["b_d1"] = dout.sum((0, 1))
    gr["W_d1"] = dout.reshape(m*k2, k1*d).T @ rows.reshape(m*k2, d)
    drows = f("dZ", dout @ p["W_d1"])
    if spec.levels == 2:
        dZ = drows.reshape(m, k2*d); gr["b_d2"] = dZ.sum(0); gr["W_d2"] = dZ.T @ Hbar
        dHbar = f("dHbar", dZ @ p["W_d2"])
    else:
        dHbar = drows.reshape(m, d)
    gr["W_o"] = dHbar.T @ A
    dA = f("dA", dHbar @ p["W_o"])
    dQ, dK, dV = np.zeros_like(Q), np.zeros_like(K), np.zeros_like(V)
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh); Pm = Ps[h]
        dO = dA[:, cs]
        dV[:, cs] = f("P", Pm).T @ dO
        dP = dO @ V[:, cs].T
        Di = (dO * A[:, cs]).sum(1, keepdims=True)
        dS = Pm * (dP - Di)
        dQ[:, cs] = f("dS", dS) @ K[:, cs] / math.sqrt(dh)
        dK[:, cs] = f("dS", dS).T @ Q[:, cs] / math.sqrt(dh)
    dQKV = f("dQKV", np.concatenate([dQ, dK, dV], 1))
    gr["W_qkv"] = dQKV.T @ Hq
    dH = dQKV @ W + (0.0 if dHo is None else dHo)
    dHb = f("dHb", dH)
    if spec.levels == 2:
        gr["b_c2"] = dH.sum(0); gr["W_c2"] = dHb.T @ Yr.reshape(m, k2*d)
        dY = f("dY", (dHb @ p["W_c2"]).reshape(m, k2, d))
    else:
        dY = dHb.reshape(m, 1, d)
    gr["b_c1"] = dY.sum((0, 1))
    gr["W_c1"] = dY.reshape(m*k2, d).T @ groups.reshape(m*k2, k1*d)
    dXc = OL.unpartition((dY @ p["W_c1"]).reshape(m, P, d), spec, L)
    dX = f("dX", dXd + dXc)
    return Xo, dX, dH, gr, H



ROUNDED = {"Y", "H", "QK", "V", "P", "A", "Hbar", "Z", "D", "Xo", "dD", "dZ", "dHbar", "dA",
           "dS", "dQKV", "dHb", "dY", "dX"}


def _rel_max(a, b):
    return float(np.abs(a - b).max() / np.sqrt(np.mean(b * b)))


def _rel_rms(a, b):
    return float(np.sqrt(np.mean((a - b) ** 2) / np.mean(b * b)))


def test_bf16_error_floor():
    spec = S.LayerSpec(batch=1, L=2048, d=128, n_heads=2, P=16, levels=2, k1=4, k2=4)
    inp = S.make_layer_inputs(spec, 1)
    p = {k: v.astype(np.float64) for k, v in inp.items()}
    X, G, dHo = p["X"][0], p["G"][0], p["dH_out"][0]
    ref = run(spec, p, X, G, dHo, set())[:4]
    exact = OL.layer_fwd(spec, inp, inp["X"])[0][0]
    np.testing.assert_allclose(ref[0], exact, rtol=1e-12, atol=1e-12)  # same math as the oracle
    got = run(spec, p, X, G, dHo, ROUNDED)[:4]
    pairs = {"X_out": (got[0], ref[0]), "dX": (got[1], ref[1]), "dH": (got[2], ref[2])}
    pairs.update({"grad " + k: (got[3][k], ref[3][k]) for k in ref[3]})
    mx = {k: _rel_max(*v) for k, v in pairs.items()}
    rr = {k: _rel_rms(*v) for k, v in pairs.items()}
    assert mx["X_out"] < 2e-2
    assert max(mx[k] for k in mx if k != "X_out") > 2e-2
    assert max(rr.values()) < 1e-2, rr
    assert max(mx.values()) < 1e-1, mx


def run_cross(spec, p, X, G, dHo, F, H_in=None):
    """``run`` for the gated cross-attention injection (Eq. inj-cross): the
    same proxy path, then token queries and gate (rounded as the stored
    [Q | gate] matrix), the proxies' keys and values, the unnormalised
    probabilities (as fed to P.V), the gated and ungated outputs and X_out;
    backward rounding at dAg, dO, dS, [dQ | d gate], [dK | dV], dHbar, the
    direct dX and the points ``run`` rounds."""
    f = lambda n, a: rb(a) if n in F else a
    L, d = X.shape; m = spec.m; nh = spec.n_heads; dh = d // nh; k1, k2, P = spec.k1, spec.k2, spec.P
    causal = spec.mode == 0
    Xb = OL.partition(X, spec)
    groups = Xb.reshape(m, k2, k1*d)
    Y = groups @ p["W_c1"].T + p["b_c1"]
    if spec.levels == 2:
        Yr = f("Y", Y); H = Yr.reshape(m, k2*d) @ p["W_c2"].T + p["b_c2"]
    else:
        H = Y.reshape(m, d); Yr = None
    if H_in is not None: H = H + H_in
    Hq = f("H", H)
    W = p["W_qkv"]
    Q, K, V = f("QK", Hq @ W[:d].T), f("QK", Hq @ W[d:2*d].T), f("V", Hq @ W[2*d:].T)
    A = np.zeros((m, d)); Ps = []
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh)
        Sm = Q[:, cs] @ K[:, cs].T / math.sqrt(dh)
        if causal: Sm = np.where(np.tril(np.ones((m, m))) > 0, Sm, -np.inf)
        Pm = np.exp(Sm - Sm.max(1, keepdims=True)); l = Pm.sum(1, keepdims=True)
        Ps.append(Pm / l)
        A[:, cs] = (f("P", Pm) @ V[:, cs]) / l
    A = f("A", A)
    Hbar = f("Hbar", A @ p["W_o"].T)
    # cross injection
    Wqa = p["W_qa"]
    Qx = f("QA", X @ Wqa[:d].T); apre = f("QA", X @ Wqa[d:].T)
    al = OL.sigmoid(apre + p["b_a"])
    Kx = f("KVx", Hbar @ p["W_kvx"][:d].T); Vx = f("KVx", Hbar @ p["W_kvx"][d:].T)
    vis = (np.arange(m)[None, :] < (np.arange(L) // P)[:, None]) if causal else np.ones((L, m), bool)
    rows = vis.any(1)
    Ax = np.zeros((L, d)); Pxs = []
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh)
        Sm = np.where(vis, Qx[:, cs] @ Kx[:, cs].T / math.sqrt(dh), -np.inf)
        mx = np.where(rows[:, None], Sm.max(1, keepdims=True), 0.0)
        Pm = np.where(vis, np.exp(Sm - mx), 0.0); l = Pm.sum(1, keepdims=True)
        ln = np.where(l > 0, l, 1.0)
        Pxs.append(Pm / ln)
        Ax[:, cs] = (f("P", Pm) @ Vx[:, cs]) / ln
    alr = np.repeat(al, dh, axis=1)
    Ag = f("Ag", alr * Ax); Axr = f("Ax", Ax)
    Xo = f("Xo", X + Ag @ p["W_ox"].T)
    # backward
    gr = {}
    gr["W_ox"] = G.T @ Ag
    dAg = f("dAg", G @ p["W_ox"])
    s = (dAg * Axr).reshape(L, nh, dh).sum(-1)
    da = s * al * (1 - al)
    gr["b_a"] = da.sum(0)
    dO = f("dOx", dAg * alr)
    Di = al * s
    dQx, dKx, dVx = np.zeros_like(Qx), np.zeros_like(Kx), np.zeros_like(Vx)
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh); Pm = Pxs[h]
        dVx[:, cs] = f("P", Pm).T @ dO[:, cs]
        dP = dO[:, cs] @ Vx[:, cs].T
        dS = Pm * (dP - Di[:, h:h+1])
        dQx[:, cs] = f("dS", dS) @ Kx[:, cs] / math.sqrt(dh)
        dKx[:, cs] = f("dS", dS).T @ Qx[:, cs] / math.sqrt(dh)
    dQA = f("dQA", np.concatenate([dQx, da], 1))
    dKV = f("dKVx", np.concatenate([dKx, dVx], 1))
    gr["W_qa"] = dQA.T @ X
    gr["W_kvx"] = dKV.T @ Hbar
    dHbar = f("dHbar", dKV @ p["W_kvx"])
    dXd = f("dXd", G + dQA @ Wqa)
    gr["W_o"] = dHbar.T @ A
    dA = f("dA", dHbar @ p["W_o"])
    dQ, dK, dV = np.zeros_like(Q), np.zeros_like(K), np.zeros_like(V)
    for h in range(nh):
        cs = slice(h*dh, (h+1)*dh); Pm = Ps[h]
        dOh = dA[:, cs]
        dV[:, cs] = f("P", Pm).T @ dOh
        dP = dOh @ V[:, cs].T
        Dih = (dOh * A[:, cs]).sum(1, keepdims=True)
        dS = Pm * (dP - Dih)
        dQ[:, cs] = f("dS", dS) @ K[:, cs] / math.sqrt(dh)
        dK[:, cs] = f("dS", dS).T @ Q[:, cs] / math.sqrt(dh)
    dQKV = f("dQKV", np.concatenate([dQ, dK, dV], 1))
    gr["W_qkv"] = dQKV.T @ Hq
    dH = dQKV @ W + (0.0 if dHo is None else dHo)
    dHb = f("dHb", dH)
    if spec.levels == 2:
        gr["b_c2"] = dH.sum(0); gr["W_c2"] = dHb.T @ Yr.reshape(m, k2*d)
        dY = f("dY", (dHb @ p["W_c2"]).reshape(m, k2, d))
    else:
        dY = dHb.reshape(m, 1, d)
    gr["b_c1"] = dY.sum((0, 1))
    gr["W_c1"] = dY.reshape(m*k2, d).T @ groups.reshape(m*k2, k1*d)
    dXc = OL.unpartition((dY @ p["W_c1"]).reshape(m, P, d), spec, L)
    dX = f("dX", dXd + dXc)
    return Xo, dX, dH, gr, H

CROSS_ROUNDED = ROUNDED | {"QA", "KVx", "Ag", "Ax", "dAg", "dOx", "dQA", "dKVx", "dXd"}


def test_bf16_error_floor_cross_injection():
    """The cross injection's floor is higher: every token's gradient reaches
    the proxies through the cross-attention, and the proxy path below it
    compounds that.  For a P = 64 two-level layer (d = 128) the RMS floor of
    dH, dX and the compression / Q,K,V weight gradients is 1-2e-2 and their
    max floor above 1e-1, X_out stays below 5e-2 max.  The GPU parity bar
    of this variant is RMS 4e-2, max 3e-1 for gradients (about twice the
    floor); the same emulation at d = 1024 gives RMS <= 1.7e-2 and max 0.23."""
    spec = S.LayerSpec(batch=1, L=4136, d=128, n_heads=2, P=64, levels=2, k1=8, k2=8,
                       inject=S.INJ_CROSS)
    inp = S.make_layer_inputs(spec, 1, with_h_in=True)
    p = {k: v.astype(np.float64) for k, v in inp.items()}
    X, G, dHo, H_in = p["X"][0], p["G"][0], p["dH_out"][0], p["H_in"][0]
    ref = run_cross(spec, p, X, G, dHo, set(), H_in)
    exact = OL.layer_fwd(spec, inp, inp["X"], inp["H_in"])[0][0]
    np.testing.assert_allclose(ref[0], exact, rtol=1e-10, atol=1e-10)  # same math as the oracle
    got = run_cross(spec, p, X, G, dHo, CROSS_ROUNDED, H_in)
    pairs = {"X_out": (got[0], ref[0]), "dX": (got[1], ref[1]), "dH": (got[2], ref[2])}
    pairs.update({"grad " + k: (got[3][k], ref[3][k]) for k in ref[3]})
    mx = {k: _rel_max(*v) for k, v in pairs.items()}
    rr = {k: _rel_rms(*v) for k, v in pairs.items()}
    assert mx["X_out"] < 5e-2, mx
    assert max(mx.values()) > 1e-1, mx
    assert max(rr.values()) > 1e-2 and max(rr.values()) < 2e-2, rr
    assert max(mx.values()) < 2e-1, mx


def run_stack(specs, params, X, G, F):
    """Layers composed with the H carry rule (same P), forward then backward."""
    xs, hs = [X], []
    for l, (sp, p) in enumerate(zip(specs, params)):
        carry = l > 0 and specs[l].P == specs[l - 1].P
        xo, _, _, _, h = run(sp, p, xs[-1], np.zeros_like(X), None, F, hs[-1] if carry else None)
        xs.append(xo)
        hs.append(h)
    g, dh_next, grads = G, None, {}
    for l in reversed(range(len(specs))):
        carry = l > 0 and specs[l].P == specs[l - 1].P
        nxt = l + 1 < len(specs) and specs[l + 1].P == specs[l].P
        _, g, dh, gr, _ = run(specs[l], params[l], xs[l], g, dh_next if nxt else None, F,
                              hs[l - 1] if carry else None)
        dh_next = dh
        grads[l] = gr
    return xs[-1], g, grads


STACK_RATIOS = (4, 4, 8, 16, 16)


def stack_case():
    specs = []
    for P in STACK_RATIOS:
        k1, k2 = S.default_factors(P)
        specs.append(S.LayerSpec(batch=1, L=1024, d=128, n_heads=2, P=P, levels=2, k1=k1, k2=k2))
    params = [{k: v.astype(np.float64) for k, v in S.make_layer_params(s, 70 + i).items()}
              for i, s in enumerate(specs)]
    inp = S.make_layer_inputs(specs[0], 80)
    return specs, params, inp["X"][0].astype(np.float64), inp["G"][0].astype(np.float64)


def test_bf16_error_floor_of_a_stack():
    """Through a five-layer stack with H carried between equal-P layers the
    rounding errors compound (the backward runs on forward activations that
    already drifted): dX and the weight gradients reach about 4e-2 RMS and
    5e-1 max relative error.  The stack test's bar -- RMS 1e-1, max 1 for
    gradients, RMS 3e-2 for X_out -- is about twice this floor; a wrong carry
    rule moves whole tensors by O(1) and still fails it."""
    specs, params, X, G = stack_case()
    ref = run_stack(specs, params, X, G, set())
    got = run_stack(specs, params, X, G, ROUNDED)
    assert _rel_rms(got[0], ref[0]) < 1.5e-2
    assert 2e-2 < _rel_rms(got[1], ref[1]) < 5e-2
    assert _rel_max(got[1], ref[1]) < 6e-1
    for l in got[2]:
        for k in ("W_c1", "W_d1", "W_qkv"):
            assert _rel_rms(got[2][l][k], ref[2][l][k]) < 5e-2
