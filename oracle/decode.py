"""Float64 oracle of the proxy KV-cache decode step and block append.

TEST INFRASTRUCTURE ONLY (see the package docstring).

Decode (Eq. llm-cross, Eq. llm-gate, Sec. 3.8), per sequence b and head h:
  q, k, v = W_q x, W_k x, W_v x; (x, k, v) go to open slot n_o;
  A_x = softmax over the open block's slots 0..n_o (the new token included)
        of q.k_j/sqrt(dh), times v_j  -- the causal self-attention of the
        generation region;
  A_h = softmax over cached proxies 0..n_p-1 of q.K_proxy_j/sqrt(dh), times
        V_proxy_j  -- a separate softmax (zero when n_p = 0);
  alpha = sigmoid(W_a2 SiLU(W_a1 RMSNorm(x) + b_a1) + b_a2), one per head;
  A = A_x + alpha_h A_h;  y = x + W_o A;  n_o += 1.
Readings: RMSNorm has eps 1e-6 and a learnable weight; the alpha MLP's hidden
width is d/8 (parity unpinned: the paper gives no width); no FFN.

Append (Sec. 3.8: once the generation region holds P new tokens, their block
is compressed and appended to the cache): the P open-block features are
compressed exactly like a layer's block (Eq.
compress-linear / Eq. factor-cascade), H = H_in + c (Eq. proxy-res), and the
proxy's key and value rows W_kh H, W_vh H are written at cache row n_p;
n_p += 1, n_o = 0.

Prefill (Sec. 3.8: the prefill stage compresses the historical blocks and
caches only their proxies): a history of L tokens gives m = floor(L / P)
complete blocks, each compressed and projected as an append does, and the
r = L - m P remaining tokens fill the open block with their features and the
decode step's keys W_k x and values W_v x; n_p = m, n_o = r.
"""
from __future__ import annotations

import math

import numpy as np

RMS_EPS = 1e-6


def _f64(a):
    return np.asarray(a, dtype=np.float64)


def _sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def _softmax_attend(q, Kr, Vr, scale):
    """softmax(Kr q * scale) @ Vr for one head; zero when there are no rows."""
    if Kr.shape[0] == 0:
        return np.zeros(Vr.shape[1])
    s = (Kr @ q) * scale
    e = np.exp(s - s.max())
    return (e / e.sum()) @ Vr


def rmsnorm(x, w):
    return x / np.sqrt((x * x).mean() + RMS_EPS) * w


def alpha_gate(x, prm):
    """alpha = MLP_alpha(RMSNorm(x)) with a sigmoid output, one value per head."""
    r = rmsnorm(x, _f64(prm["rms_w"]))
    a1 = _f64(prm["W_a1"]) @ r + _f64(prm["b_a1"])
    u = a1 * _sigmoid(a1)
    return _sigmoid(_f64(prm["W_a2"]) @ u + _f64(prm["b_a2"]))


def decode_step(spec, prm, state, return_parts=False):
    """One decode step for every sequence.  ``state`` holds K_proxy, V_proxy
    [B, cap, d], X_open, K_open, V_open [B, P, d], n_proxy, n_open [B] and the
    new token x [B, d].  Returns (y [B, d], new_state) where new_state has the
    token written at its open slot and n_open advanced."""
    B, d = state["x"].shape
    nh, dh = spec.n_heads, spec.d // spec.n_heads
    scale = 1.0 / math.sqrt(dh)
    W = _f64(prm["W_qkv"])
    new = {k: np.array(v, copy=True) for k, v in state.items()}
    new["X_open"] = _f64(new["X_open"])
    new["K_open"] = _f64(new["K_open"])
    new["V_open"] = _f64(new["V_open"])
    y = np.zeros((B, d))
    parts = []
    for b in range(B):
        x = _f64(state["x"][b])
        q, k, v = W[:d] @ x, W[d:2 * d] @ x, W[2 * d:] @ x
        no, npx = int(state["n_open"][b]), int(state["n_proxy"][b])
        new["X_open"][b, no] = x
        new["K_open"][b, no] = k
        new["V_open"][b, no] = v
        Ko, Vo = new["K_open"][b, :no + 1], new["V_open"][b, :no + 1]
        Kp, Vp = _f64(state["K_proxy"][b, :npx]), _f64(state["V_proxy"][b, :npx])
        Ax, Ah = np.zeros(d), np.zeros(d)
        for h in range(nh):
            cs = slice(h * dh, (h + 1) * dh)
            Ax[cs] = _softmax_attend(q[cs], Ko[:, cs], Vo[:, cs], scale)
            Ah[cs] = _softmax_attend(q[cs], Kp[:, cs], Vp[:, cs], scale)
        alpha = alpha_gate(x, prm)
        A = Ax + np.repeat(alpha, dh) * Ah
        y[b] = x + _f64(prm["W_o"]) @ A
        parts.append(dict(q=q, k=k, v=v, Ax=Ax, Ah=Ah, alpha=alpha))
        new["n_open"][b] = no + 1
    return (y, new, parts) if return_parts else (y, new)


def compress_block(Xblk, prm, spec):
    """c = C(X_blk) for one block [P, d] (Eq. compress-linear; with two levels
    Eq. factor-cascade: k2 groups of k1 tokens -> rows -> one proxy)."""
    P, d = Xblk.shape
    k1, k2 = spec.k1, spec.k2
    Y = Xblk.reshape(k2, k1 * d) @ _f64(prm["W_c1"]).T + _f64(prm["b_c1"])
    if spec.levels == 1:
        return Y.reshape(d)
    return _f64(prm["W_c2"]) @ Y.reshape(k2 * d) + _f64(prm["b_c2"])


def kv_append(spec, prm, state, H_in=None):
    """Compress each sequence's full open block into a proxy and append its
    key/value rows to the cache.  Returns the new state."""
    B = state["n_open"].shape[0]
    d = spec.d
    new = {k: np.array(v, copy=True) for k, v in state.items()}
    new["K_proxy"] = _f64(new["K_proxy"])
    new["V_proxy"] = _f64(new["V_proxy"])
    Wkv = _f64(prm["W_kvh"])
    for b in range(B):
        c = compress_block(_f64(state["X_open"][b]), prm, spec)
        H = c if H_in is None else _f64(H_in[b]) + c
        npx = int(state["n_proxy"][b])
        new["K_proxy"][b, npx] = Wkv[:d] @ H
        new["V_proxy"][b, npx] = Wkv[d:] @ H
        new["n_proxy"][b] = npx + 1
        new["n_open"][b] = 0
    return new


def kv_prefill(spec, prm, X_hist, H_in=None):
    """Cache state after prefilling from a history X_hist [B, L, d]: all
    complete blocks compressed at once (the blocks' rows of k1 tokens through
    W_c1, their k2 rows through W_c2 with two levels), H = H_in + C, proxy
    rows W_kh H / W_vh H; the remaining tokens' features, W_k x and W_v x in
    the open block.  H_in [B, ceil(L / P), d] (a layer's proxy stream; the
    partial block's row unused) or None.  Rows past n_proxy / n_open are
    zero."""
    X = _f64(X_hist)
    B, L, d = X.shape
    P, k1, k2 = spec.P, spec.k1, spec.k2
    m, r = L // P, L % P
    Y = X[:, :m * P].reshape(B * m * k2, k1 * d) @ _f64(prm["W_c1"]).T + _f64(prm["b_c1"])
    if spec.levels == 1:
        C = Y.reshape(B, m, d)
    else:
        C = (Y.reshape(B * m, k2 * d) @ _f64(prm["W_c2"]).T + _f64(prm["b_c2"])).reshape(B, m, d)
    H = C if H_in is None else C + _f64(H_in)[:, :m]
    Wkv, Wqkv = _f64(prm["W_kvh"]), _f64(prm["W_qkv"])
    st = {k: np.zeros((B, spec.capacity, d)) for k in ("K_proxy", "V_proxy")}
    st.update({k: np.zeros((B, P, d)) for k in ("X_open", "K_open", "V_open")})
    st["K_proxy"][:, :m] = H @ Wkv[:d].T
    st["V_proxy"][:, :m] = H @ Wkv[d:].T
    Xr = X[:, m * P:]
    st["X_open"][:, :r] = Xr
    st["K_open"][:, :r] = Xr @ Wqkv[d:2 * d].T
    st["V_open"][:, :r] = Xr @ Wqkv[2 * d:].T
    st["n_proxy"] = np.full(B, m, dtype=np.int32)
    st["n_open"] = np.full(B, r, dtype=np.int32)
    return st
