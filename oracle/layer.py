"""Float64 oracle of one ProxyFormer layer (Alg. 1), forward and backward.

TEST INFRASTRUCTURE ONLY (see the package docstring): a plain restatement of
the paper's equations, one step per function, no blocking, fusion or
reordering.  Library matmuls serve as steps.

Readings of the paper taken here (each is a descriptor flag of the library):
  * Causal 1D routing: the tokens of block i receive the decompression of the
    interacted proxy i-1; block 0 receives zero.  (Proxy i summarises tokens
    that come after the early tokens of block i, so this shift is the reading
    under which a token never sees a later token; it also matches the decode
    rule that only completed blocks are cached, Sec. 3.8.)
  * F is standard multi-head attention with an output projection and no
    biases; no norm inside F for 1D; the 2D layer applies adaptive LayerNorm
    (timestep-conditioned scale/shift) to the proxies before attention, the
    only place conditions touch the proxies (Sec. 3.9).
  * Gate g(X, D) = w_x*X + w_dlt*D + b_g per channel (Eq. inj-gate).
  * H carried to the next layer is the pre-interaction H (Alg. 1 returns H).
  * Two-level cascade: no nonlinearity between levels, biases at each level.
  * Affine injection (Eq. inj-affine): s and t are the two halves of a
    2*P*d-wide decompression (token p takes [s | t] from columns
    [2pd, 2pd+d) and [2pd+d, 2(p+1)d)); Norm is LayerNorm without affine,
    biased variance, eps 1e-6.
  * L % P != 0: the last block is zero-padded for compression (m = ceil(L/P)).
  * Proxy interaction F (Sec. 3.4): attention (Eq. proxy-attn), identity
    (Hbar = H) or a single-proxy MLP Hbar = W_m2 SiLU(W_m1 H + b_m1) + b_m2 of
    hidden width 4d; attention may rotate the proxies' queries and keys by
    their index (RoPE, base 10000, pairs (2j, 2j+1) of each head).
  * Temporal-distance ratios (Sec. 3.6): a causal sequence split into
    segments with their own block size (coarse blocks for distant history),
    each with its own compression / decompression weights; one causal
    attention over all proxies in time order; a block receives the proxy
    just before it in time, decompressed by its own segment's weights.
  * Widths: tokens are d_fine wide and proxies d wide (d_fine = d unless the
    spec says otherwise, the asymmetric history stream of the language
    model); both compression levels output d, both decompression levels read d.
  * Cross-attention injection (Eq. inj-cross) in its gated form, the way the
    language model uses it (Eq. llm-cross / llm-gate): every token queries,
    per head, the interacted proxies it may see (causal: proxies of earlier
    blocks only, the same one-block shift as above; bidirectional: all of
    them); a per-head linear gate alpha = sigmoid(W_a x + b_a) scales each
    head's result; X_out = X + W_ox (alpha * A).  W_qa stacks the token-query
    projection [d, d] over the gate's rows [heads, d]; W_kvx maps proxies to
    the injection's keys and values.  No decompression is used.
"""
from __future__ import annotations

import math
from typing import Dict, Optional

import numpy as np

CAUSAL_1D, BIDIR_1D, BIDIR_2D = 0, 1, 2
F_ATTENTION, F_IDENTITY, F_MLP = 0, 1, 2
ROPE_BASE = 10000.0
INJ_ADD, INJ_GATED, INJ_AFFINE, INJ_CROSS = 0, 1, 2, 3
LN_EPS = 1e-6
TEMB_DIM = 256


def _f64(a):
    return None if a is None else np.asarray(a, dtype=np.float64)


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


# ---------------------------------------------------------------- partition
def partition(X, spec):
    """Eq. partition (Sec. 3.2, partitioning): split one sequence X [L, d]
    into m = ceil(L/P) blocks X_i [P, d].  1D: contiguous non-overlapping
    blocks, the last zero-padded.  2D: p x p spatial patches of the
    grid_h x grid_w raster, patches in raster order, tokens inside a patch in
    raster order (py, px)."""
    L, d = X.shape
    P = spec.P
    if spec.mode == BIDIR_2D:
        p, gh, gw = spec.patch, spec.grid_h, spec.grid_w
        g = X.reshape(gh // p, p, gw // p, p, d)          # (by, py, bx, px, ch)
        return g.transpose(0, 2, 1, 3, 4).reshape(-1, P, d)  # (by*bx, py*px, ch)
    m = -(-L // P)
    Xp = np.zeros((m * P, d))
    Xp[:L] = X
    return Xp.reshape(m, P, d)


def unpartition(blocks, spec, L):
    """Inverse of ``partition``: per-token array [L, w] from [m, P, w]."""
    m, P, w = blocks.shape
    if spec.mode == BIDIR_2D:
        p, gh, gw = spec.patch, spec.grid_h, spec.grid_w
        g = blocks.reshape(gh // p, gw // p, p, p, w).transpose(0, 2, 1, 3, 4)
        return g.reshape(gh * gw, w)
    return blocks.reshape(m * P, w)[:L]


# -------------------------------------------------------------- compression
def compress(Xb, prm, spec):
    """Eq. compress-linear and Eq. factor-cascade: c_i = Proj(Flatten(X_i)).

    Flatten is token-major (index p*d_fine + ch).  Two levels: level 1 groups
    the P tokens into k2 consecutive groups of k1 and projects each group's
    k1*d_fine vector to d (y_{i,a}); level 2 concatenates the k2 rows and
    projects the k2*d vector to d.  Returns C [m, d] and the level-1 rows Y
    [m, k2, d]."""
    m, P, df = Xb.shape
    k1, k2, d = spec.k1, spec.k2, spec.d
    groups = Xb.reshape(m, k2, k1 * df)                    # vec of each group
    Y = groups @ _f64(prm["W_c1"]).T + _f64(prm["b_c1"])   # [m, k2, d]
    if spec.levels == 1:
        return Y.reshape(m, d), None
    C = Y.reshape(m, k2 * d) @ _f64(prm["W_c2"]).T + _f64(prm["b_c2"])
    return C, Y


def decompress(Hbar, prm, spec):
    """Eq. decompress-linear and Eq. factor-dec: D_i = Unflatten(Proj_up(Hbar_i)).

    Two levels run in the opposite order: level 2 maps the proxy to k2 rows of
    width d, level 1 maps each row to k1 tokens.  Output [m, P, w] with w =
    d_fine, or w = 2d for affine injection ([s | t] per token)."""
    m, d = Hbar.shape
    k1, k2 = spec.k1, spec.k2
    if spec.levels == 2:
        Z = Hbar @ _f64(prm["W_d2"]).T + _f64(prm["b_d2"])  # [m, k2*d]
        rows = Z.reshape(m, k2, d)
    else:
        Z = None
        rows = Hbar.reshape(m, 1, d)
    out = rows @ _f64(prm["W_d1"]).T + _f64(prm["b_d1"])  # [m, k2, k1*w]
    w = out.shape[-1] // k1
    return out.reshape(m, k1 * k2, w), Z


# ---------------------------------------------------------------- attention
def proxy_mask(m, spec):
    """The mask M of Eq. proxy-attn as a boolean [m, m] matrix of visible
    (query, key) pairs: proxy i sees j <= i in the autoregressive 1D mode and
    every proxy otherwise."""
    if spec.mode == CAUSAL_1D:
        return np.tril(np.ones((m, m), dtype=bool))
    return np.ones((m, m), dtype=bool)


def _probs(Qh, Kh, vis, scale):
    """softmax(Q K^T * scale + M) row by row, M = -inf where ``vis`` is
    False, with each row's maximum subtracted (every row sees its own key)."""
    S = np.where(vis, (Qh @ Kh.T) * scale, -np.inf)
    E = np.exp(S - S.max(1, keepdims=True))
    return E / E.sum(1, keepdims=True)


def rope(Z, nh, inverse=False):
    """Rotary position embedding of rows Z [m, d] by their index i: within
    each head, the pair (2j, 2j+1) turns by the angle i * ROPE_BASE^(-2j/dh)
    (backwards when ``inverse``, the transpose of the rotation)."""
    m, d = Z.shape
    dh = d // nh
    j = np.arange(dh // 2)
    ang = np.arange(m)[:, None] * ROPE_BASE ** (-2.0 * j / dh)[None, :]  # [m, dh/2]
    c, s = np.cos(ang), np.sin(ang)
    if inverse:
        s = -s
    out = np.empty_like(Z)
    for h in range(nh):
        a = Z[:, h * dh:(h + 1) * dh:2]
        b = Z[:, h * dh + 1:(h + 1) * dh:2]
        out[:, h * dh:(h + 1) * dh:2] = a * c - b * s
        out[:, h * dh + 1:(h + 1) * dh:2] = a * s + b * c
    return out


def silu_grad(u):
    sg = sigmoid(u)
    return sg * (1.0 + u * (1.0 - sg))


def interact(Hq, prm, spec):
    """The proxy interaction F (Sec. 3.4): identity, single-proxy MLP, or
    attention (below)."""
    f = getattr(spec, "interact", F_ATTENTION)
    if f == F_IDENTITY:
        return Hq.copy(), {}
    if f == F_MLP:
        U = Hq @ _f64(prm["W_m1"]).T + _f64(prm["b_m1"])
        Am = silu(U)
        return Am @ _f64(prm["W_m2"]).T + _f64(prm["b_m2"]), dict(U=U, Am=Am)
    return attention(Hq, prm, spec)


def interact_bwd(dHbar, c, prm, spec, grads):
    """Backward of ``interact``: dHq, adding the interaction's weight gradients."""
    f = getattr(spec, "interact", F_ATTENTION)
    if f == F_IDENTITY:
        return dHbar
    if f == F_MLP:
        grads["W_m2"] += dHbar.T @ c["Am"]
        grads["b_m2"] += dHbar.sum(0)
        dU = (dHbar @ _f64(prm["W_m2"])) * silu_grad(c["U"])
        grads["W_m1"] += dU.T @ c["Hq"]
        grads["b_m1"] += dU.sum(0)
        return dU @ _f64(prm["W_m1"])
    grads["W_o"] += dHbar.T @ c["A"]
    dA = dHbar @ _f64(prm["W_o"])
    dQ, dK, dV = attention_bwd(dA, c, spec)
    if getattr(spec, "rope", 0):                          # back through the rotation
        dQ, dK = rope(dQ, spec.n_heads, True), rope(dK, spec.n_heads, True)
    dQKV = np.concatenate([dQ, dK, dV], axis=1)
    grads["W_qkv"] += dQKV.T @ c["Hq"]
    return dQKV @ _f64(prm["W_qkv"])


def attention(Hq, prm, spec):
    """Eq. proxy-attn: Hbar = softmax(Q K^T / sqrt(dh) + M) V per head, then
    the output projection.  M is the causal mask (proxy i sees j <= i) for the
    autoregressive 1D mode and zero otherwise; each head's m x m probability
    matrix is formed whole.  With RoPE, Q and K are rotated by the proxy index
    first."""
    m, d = Hq.shape
    nh, dh = spec.n_heads, d // spec.n_heads
    W = _f64(prm["W_qkv"])
    Q, K, V = Hq @ W[:d].T, Hq @ W[d:2 * d].T, Hq @ W[2 * d:].T
    if getattr(spec, "rope", 0):
        Q, K = rope(Q, nh), rope(K, nh)
    A = np.zeros((m, d))
    scale = 1.0 / math.sqrt(dh)
    vis = proxy_mask(m, spec)
    for h in range(nh):
        cs = slice(h * dh, (h + 1) * dh)
        A[:, cs] = _probs(Q[:, cs], K[:, cs], vis, scale) @ V[:, cs]
    Hbar = A @ _f64(prm["W_o"]).T
    return Hbar, dict(Q=Q, K=K, V=V, A=A)


def attention_bwd(dA, c, spec):
    """Backward of the attention core per head: with P the probability
    matrix, dV = P^T dO, dP = dO V^T, dS = P * (dP - rowsum(P * dP)),
    dQ = scale dS K, dK = scale dS^T Q."""
    Q, K, V = c["Q"], c["K"], c["V"]
    m, d = Q.shape
    nh, dh = spec.n_heads, d // spec.n_heads
    scale = 1.0 / math.sqrt(dh)
    vis = proxy_mask(m, spec)
    dQ, dK, dV = np.zeros_like(Q), np.zeros_like(K), np.zeros_like(V)
    for h in range(nh):
        cs = slice(h * dh, (h + 1) * dh)
        Pm = _probs(Q[:, cs], K[:, cs], vis, scale)
        dO = dA[:, cs]
        dV[:, cs] = Pm.T @ dO
        dP = dO @ V[:, cs].T
        dS = Pm * (dP - (Pm * dP).sum(1, keepdims=True))
        dQ[:, cs] = scale * (dS @ K[:, cs])
        dK[:, cs] = scale * (dS.T @ Q[:, cs])
    return dQ, dK, dV


# ------------------------------------------------- cross-attention injection
def _cross_visible(L, m, spec):
    """[L, m] mask of the proxies each token may read: those of earlier
    blocks (causal, proxy j < t // P), else all."""
    if spec.mode == CAUSAL_1D:
        return np.arange(m)[None, :] < (np.arange(L) // spec.P)[:, None]
    return np.ones((L, m), dtype=bool)


def _cross_probs(Qh, Kh, vis, scale):
    """Row-wise softmax of the scores Q K^T * scale over the visible
    proxies (the row maximum subtracted); a row that sees none is zero."""
    S = np.where(vis, (Qh @ Kh.T) * scale, -np.inf)
    mx = np.where(vis.any(1), S.max(1, initial=-np.inf), 0.0)
    E = np.where(vis, np.exp(S - mx[:, None]), 0.0)
    l = E.sum(1)
    return E / np.where(l > 0, l, 1.0)[:, None]


def cross_inject(X, Hbar, prm, spec):
    """Gated Eq. inj-cross over one sequence: Q = X W_q^T, alpha = sigmoid(
    X W_a^T + b_a) per head, K, V = Hbar W_k^T, Hbar W_v^T; row t of head h
    is the softmax over its visible proxies (a token that sees none gets 0);
    X_out = X + (alpha * A) W_ox^T."""
    L, d = X.shape
    m = Hbar.shape[0]
    nh, dh = spec.n_heads, d // spec.n_heads
    Wqa, Wkv = _f64(prm["W_qa"]), _f64(prm["W_kvx"])
    Q = X @ Wqa[:d].T
    alpha = sigmoid(X @ Wqa[d:].T + _f64(prm["b_a"]))           # [L, heads]
    K, V = Hbar @ Wkv[:d].T, Hbar @ Wkv[d:].T
    A = np.zeros((L, d))
    scale = 1.0 / math.sqrt(dh)
    vis = _cross_visible(L, m, spec)
    for h in range(nh):
        cs = slice(h * dh, (h + 1) * dh)
        A[:, cs] = _cross_probs(Q[:, cs], K[:, cs], vis, scale) @ V[:, cs]
    Ag = A * np.repeat(alpha, dh, axis=1)
    Xo = X + Ag @ _f64(prm["W_ox"]).T
    return Xo, dict(Qx=Q, Kx=K, Vx=V, Ax=A, alpha=alpha, Ag=Ag)


def cross_inject_bwd(G, X, Hbar, c, prm, spec, grads):
    """Chain rule through ``cross_inject``: returns (dX, dHbar) and adds the
    gradients of W_ox, W_qa, b_a and W_kvx to ``grads``."""
    L, d = X.shape
    m = Hbar.shape[0]
    nh, dh = spec.n_heads, d // spec.n_heads
    scale = 1.0 / math.sqrt(dh)
    Q, K, V, A, alpha = c["Qx"], c["Kx"], c["Vx"], c["Ax"], c["alpha"]
    grads["W_ox"] += G.T @ c["Ag"]
    dAg = G @ _f64(prm["W_ox"])
    s = (dAg * A).reshape(L, nh, dh).sum(-1)                     # dL/dalpha
    da = s * alpha * (1.0 - alpha)                                # through the sigmoid
    dA = dAg * np.repeat(alpha, dh, axis=1)
    dQ, dK, dV = np.zeros_like(Q), np.zeros_like(K), np.zeros_like(V)
    vis = _cross_visible(L, m, spec)
    for h in range(nh):     # with p the probabilities of each row: dV = p^T dO,
        cs = slice(h * dh, (h + 1) * dh)        # dS = p * (dp - <p, dp>), dp = dO V^T
        p = _cross_probs(Q[:, cs], K[:, cs], vis, scale)
        dO = dA[:, cs]
        dV[:, cs] = p.T @ dO
        dp = dO @ V[:, cs].T
        dS = p * (dp - (p * dp).sum(1, keepdims=True))
        dQ[:, cs] = scale * (dS @ K[:, cs])
        dK[:, cs] = scale * (dS.T @ Q[:, cs])
    dQA = np.concatenate([dQ, da], axis=1)
    Wqa, Wkv = _f64(prm["W_qa"]), _f64(prm["W_kvx"])
    grads["W_qa"] += dQA.T @ X
    grads["b_a"] += da.sum(0)
    dKV = np.concatenate([dK, dV], axis=1)
    grads["W_kvx"] += dKV.T @ Hbar
    return G + dQA @ Wqa, dKV @ Wkv


# ----------------------------------------------------------- 2D conditioning
def timestep_embedding(t):
    """Sinusoidal embedding of the flow-matching time t (this library's own
    definition; the paper fixes none): e_k = cos(1000 t w_k),
    e_{128+k} = sin(1000 t w_k), w_k = 10000^(-k/128), k < 128."""
    half = TEMB_DIM // 2
    w = 10000.0 ** (-np.arange(half) / half)
    a = 1000.0 * float(t) * w
    return np.concatenate([np.cos(a), np.sin(a)])


def layernorm(x):
    """LayerNorm over the last axis, no affine, biased variance, eps 1e-6."""
    mu = x.mean(-1, keepdims=True)
    var = ((x - mu) ** 2).mean(-1, keepdims=True)
    return (x - mu) / np.sqrt(var + LN_EPS), mu, np.sqrt(var + LN_EPS)


def silu(x):
    return x * sigmoid(x)


def adaln_params(t, prm):
    """Timestep conditioning of the proxy stream (Sec. 3.9: conditions touch
    only the proxies): u = SiLU(W_t1 e(t) + b_t1), [gamma | beta] = W_t2 u + b_t2."""
    e = timestep_embedding(t)
    a1 = _f64(prm["W_t1"]) @ e + _f64(prm["b_t1"])
    u = silu(a1)
    gb = _f64(prm["W_t2"]) @ u + _f64(prm["b_t2"])
    d = gb.shape[0] // 2
    return gb[:d], gb[d:], dict(e=e, a1=a1, u=u)


# ------------------------------------------------------------------ forward
def _fwd_one(spec, prm, X, H_in, t):
    L, d = X.shape
    Xb = partition(X, spec)                                   # Eq. partition
    C, Y = compress(Xb, prm, spec)                            # Eq. compress-linear
    H = C if H_in is None else H_in + C                       # Eq. proxy-res
    cache = dict(Xb=Xb, Y=Y, H=H)
    Hq = H
    if spec.mode == BIDIR_2D:                                 # Sec. 3.9
        gamma, beta, tc = adaln_params(t, prm)
        nH, muH, sdH = layernorm(H)
        Hq = (1.0 + gamma) * nH + beta
        cache.update(gamma=gamma, beta=beta, tc=tc, nH=nH, sdH=sdH)
    Hbar, ac = interact(Hq, prm, spec)                        # F: Eq. proxy-attn, ...
    cache.update(Hq=Hq, Hbar=Hbar, **ac)
    if spec.inject == INJ_CROSS:                              # Eq. inj-cross (gated)
        Xo, cc = cross_inject(X, Hbar, prm, spec)
        cache.update(cc)
        return Xo, H, cache
    D, Z = decompress(Hbar, prm, spec)                        # Eq. decompress-linear
    cache.update(Z=Z, D=D)
    m = Xb.shape[0]
    if spec.mode == CAUSAL_1D:                                # routing shift
        Dr = np.zeros_like(D)
        Dr[1:] = D[:-1]
    else:
        Dr = D
    Dt = unpartition(Dr, spec, L)                             # per-token update
    cache["Dt"] = Dt
    if spec.inject == INJ_ADD:                                # Eq. inj-add
        Xo = X + Dt
    elif spec.inject == INJ_GATED:                            # Eq. inj-gate
        g = _f64(prm["w_x"]) * X + _f64(prm["w_dlt"]) * Dt + _f64(prm["b_g"])
        sg = sigmoid(g)
        Xo = X + sg * Dt
        cache["sg"] = sg
    else:                                                     # Eq. inj-affine
        s, tau = Dt[:, :d], Dt[:, d:]
        nX, muX, sdX = layernorm(X)
        Xo = (1.0 + s) * nX + tau
        cache.update(nX=nX, sdX=sdX)
    return Xo, H, cache


def layer_fwd(spec, prm: Dict[str, np.ndarray], X, H_in=None, t=None,
              return_cache: bool = False):
    """Alg. 1 over a batch: X [B, L, d] -> (X_out [B, L, d], H_out [B, m, d])."""
    X = _f64(X)
    outs, hs, caches = [], [], []
    for b in range(X.shape[0]):
        hin = None if H_in is None else _f64(H_in[b])
        tb = None if t is None else float(t[b])
        Xo, H, c = _fwd_one(spec, prm, X[b], hin, tb)
        outs.append(Xo)
        hs.append(H)
        caches.append(c)
    res = (np.stack(outs), np.stack(hs))
    return res + (caches,) if return_cache else res


# ----------------------------------------------------------------- backward
def _layernorm_bwd(dn, n, sd):
    """Gradient through n = (x - mean)/sd with sd = sqrt(var + eps)."""
    return (dn - dn.mean(-1, keepdims=True)
            - n * (dn * n).mean(-1, keepdims=True)) / sd


def _inject_decompress_bwd(spec, prm, X, c, G, grads):
    """Backward of the decompression, routing and Eq. inj-add / inj-gate /
    inj-affine: returns (dX direct, dHbar)."""
    L, d = X.shape                                             # token width
    dp = spec.d                                                # proxy width
    m = c["Xb"].shape[0]
    P, k1, k2 = spec.P, spec.k1, spec.k2
    Dt = c["Dt"]
    if spec.inject == INJ_ADD:
        dX = G.copy()
        dDt = G.copy()
    elif spec.inject == INJ_GATED:
        sg = c["sg"]
        ds = G * Dt * sg * (1.0 - sg)                          # dL/dg
        dX = G + ds * _f64(prm["w_x"])
        dDt = G * sg + ds * _f64(prm["w_dlt"])
        grads["w_x"] += (ds * X).sum(0)
        grads["w_dlt"] += (ds * Dt).sum(0)
        grads["b_g"] += ds.sum(0)
    else:
        nX, sdX = c["nX"], c["sdX"]
        s = Dt[:, :d]
        dDt = np.concatenate([G * nX, G], axis=1)
        dX = _layernorm_bwd(G * (1.0 + s), nX, sdX)
    # routing
    w = dDt.shape[1]
    if spec.mode == BIDIR_2D:
        dDr = partition_w(dDt, spec)
    else:
        pad = np.zeros((m * P, w))
        pad[:L] = dDt
        dDr = pad.reshape(m, P, w)
    if spec.mode == CAUSAL_1D:
        dD = np.zeros_like(dDr)
        dD[:-1] = dDr[1:]
    else:
        dD = dDr
    # decompression
    dout = dD.reshape(m, k2, k1 * w)
    grads["b_d1"] += dout.sum((0, 1))
    rows = c["Z"].reshape(m, k2, dp) if spec.levels == 2 else c["Hbar"].reshape(m, 1, dp)
    grads["W_d1"] += dout.reshape(m * k2, k1 * w).T @ rows.reshape(m * k2, dp)
    drows = dout @ _f64(prm["W_d1"])                           # [m, k2, dp]
    if spec.levels == 2:
        dZ = drows.reshape(m, k2 * dp)
        grads["b_d2"] += dZ.sum(0)
        grads["W_d2"] += dZ.T @ c["Hbar"]
        dHbar = dZ @ _f64(prm["W_d2"])
    else:
        dHbar = drows.reshape(m, dp)
    return dX, dHbar


def _bwd_one(spec, prm, X, c, G, dH_out, grads):
    L, df = X.shape                                            # token width
    d = spec.d                                                 # proxy width
    m = c["Xb"].shape[0]
    P, k1, k2 = spec.P, spec.k1, spec.k2
    if spec.inject == INJ_CROSS:
        dX, dHbar = cross_inject_bwd(G, X, c["Hbar"], c, prm, spec, grads)
    else:
        dX, dHbar = _inject_decompress_bwd(spec, prm, X, c, G, grads)
    # proxy interaction
    dHq = interact_bwd(dHbar, c, prm, spec, grads)
    if spec.mode == BIDIR_2D:
        gamma = c["gamma"]
        nH, sdH = c["nH"], c["sdH"]
        dgamma = (dHq * nH).sum(0)
        dbeta = dHq.sum(0)
        dH = _layernorm_bwd(dHq * (1.0 + gamma), nH, sdH)
        tc = c["tc"]
        dgb = np.concatenate([dgamma, dbeta])
        grads["b_t2"] += dgb
        grads["W_t2"] += np.outer(dgb, tc["u"])
        du = _f64(prm["W_t2"]).T @ dgb
        sa = sigmoid(tc["a1"])
        da1 = du * (sa * (1.0 + tc["a1"] * (1.0 - sa)))
        grads["b_t1"] += da1
        grads["W_t1"] += np.outer(da1, tc["e"])
    else:
        dH = dHq
    if dH_out is not None:
        dH = dH + dH_out
    dH_in = dH.copy()
    # compression
    dC = dH
    if spec.levels == 2:
        grads["b_c2"] += dC.sum(0)
        grads["W_c2"] += dC.T @ c["Y"].reshape(m, k2 * d)
        dY = (dC @ _f64(prm["W_c2"])).reshape(m, k2, d)
    else:
        dY = dC.reshape(m, 1, d)
    grads["b_c1"] += dY.sum((0, 1))
    groups = c["Xb"].reshape(m, k2, k1 * df)
    grads["W_c1"] += dY.reshape(m * k2, d).T @ groups.reshape(m * k2, k1 * df)
    dgroups = dY @ _f64(prm["W_c1"])                          # [m, k2, k1*df]
    dXc = unpartition(dgroups.reshape(m, P, df), spec, L)
    return dX + dXc, dH_in


# ------------------------------------------- temporal-distance ratios (Sec. 3.6)
def _seg_spec(spec, seg):
    """The single-ratio view of one segment: seg = (L, P) or, with two
    levels, (L, P, k1, k2)."""
    import dataclasses
    L, P = seg[0], seg[1]
    if spec.levels == 2:
        return dataclasses.replace(spec, L=L, P=P, k1=seg[2], k2=seg[3])
    return dataclasses.replace(spec, L=L, P=P, k1=0, k2=0)


def layer_fwd_segments(spec, segs, seg_prm, prm, X):
    """A causal 1D layer whose blocks grow coarser with temporal distance
    (Sec. 3.6): segs = [(L_s, P_s[, k1_s, k2_s]), ...] in time order (L_s a
    multiple of P_s except the last), X [sum L_s, d] one sequence.  Segment s compresses its
    blocks with its own weights seg_prm[s] (W_c1, b_c1[, W_c2, b_c2]); all
    proxies, in time order, share one causal attention (prm: W_qkv, W_o); the
    block with global proxy index g receives the interacted proxy g - 1
    decompressed by its own segment's weights (W_d*, b_d*), block 0 nothing;
    gated injection with the shared gate vectors in prm.  Returns X_out and
    the cache ``layer_bwd_segments`` reads."""
    X = _f64(X)
    Hs, parts, off = [], [], 0
    for seg, sp in zip(segs, seg_prm):
        ss = _seg_spec(spec, seg)
        Ls = ss.L
        Xb = partition(X[off:off + Ls], ss)
        C, Y = compress(Xb, sp, ss)
        Hs.append(C)
        parts.append(dict(ss=ss, Xb=Xb, Y=Y, off=off, m=Xb.shape[0]))
        off += Ls
    H = np.concatenate(Hs)
    Hbar, ac = attention(H, prm, spec)                       # causal over all proxies
    Xo = X.copy()
    g0 = 0
    for part, sp in zip(parts, seg_prm):
        ss, m, o = part["ss"], part["m"], part["off"]
        src = np.zeros((m, Hbar.shape[1]))                   # proxy g - 1 for block g
        lo = max(g0 - 1, 0)
        src[(1 if g0 == 0 else 0):] = Hbar[lo:g0 + m - 1]
        D, Z = decompress(src, sp, ss)
        if g0 == 0:
            D[0] = 0.0                                       # block 0 receives nothing
        Dt = unpartition(D, ss, ss.L)
        Xs = X[o:o + ss.L]
        sg = sigmoid(_f64(prm["w_x"]) * Xs + _f64(prm["w_dlt"]) * Dt + _f64(prm["b_g"]))
        Xo[o:o + ss.L] = Xs + sg * Dt
        part.update(src=src, Z=Z, Dt=Dt, sg=sg, g0=g0)
        g0 += m
    return Xo, dict(parts=parts, H=H, Hbar=Hbar, **ac)


def layer_bwd_segments(spec, segs, seg_prm, prm, X, G):
    """Backward of ``layer_fwd_segments`` for one sequence: (dX, seg_grads,
    grads) with the per-segment and shared weight gradients."""
    X, G = _f64(X), _f64(G)
    _, c = layer_fwd_segments(spec, segs, seg_prm, prm, X)
    d = spec.d
    grads = {k: np.zeros(np.shape(v)) for k, v in prm.items()}
    sgr = [{k: np.zeros(np.shape(v)) for k, v in sp.items()} for sp in seg_prm]
    dX = np.zeros_like(X)
    dHbar = np.zeros_like(c["Hbar"])
    for part, sp, gr in zip(c["parts"], seg_prm, sgr):
        ss, m, o, g0 = part["ss"], part["m"], part["off"], part["g0"]
        Xs, Gs, Dt, sg = X[o:o + ss.L], G[o:o + ss.L], part["Dt"], part["sg"]
        ds = Gs * Dt * sg * (1.0 - sg)                       # through the gate
        dX[o:o + ss.L] += Gs + ds * _f64(prm["w_x"])
        dDt = Gs * sg + ds * _f64(prm["w_dlt"])
        grads["w_x"] += (ds * Xs).sum(0)
        grads["w_dlt"] += (ds * Dt).sum(0)
        grads["b_g"] += ds.sum(0)
        pad = np.zeros((m * ss.P, d))
        pad[:ss.L] = dDt
        dout = pad.reshape(m, ss.k2, ss.k1 * d)
        if g0 == 0:
            dout[0] = 0.0                                    # block 0's update was zeroed
        gr["b_d1"] += dout.sum((0, 1))
        rows = part["Z"].reshape(m, ss.k2, d) if ss.levels == 2 else part["src"].reshape(m, 1, d)
        gr["W_d1"] += dout.reshape(m * ss.k2, ss.k1 * d).T @ rows.reshape(m * ss.k2, d)
        drows = dout @ _f64(sp["W_d1"])
        if ss.levels == 2:
            dZ = drows.reshape(m, ss.k2 * d)
            gr["b_d2"] += dZ.sum(0)
            gr["W_d2"] += dZ.T @ part["src"]
            dsrc = dZ @ _f64(sp["W_d2"])
        else:
            dsrc = drows.reshape(m, d)
        lo = max(g0 - 1, 0)
        dHbar[lo:g0 + m - 1] += dsrc[(1 if g0 == 0 else 0):]
    cc = dict(Q=c["Q"], K=c["K"], V=c["V"], A=c["A"], Hq=c["H"])
    dH = interact_bwd(dHbar, cc, prm, spec, grads)
    g0 = 0
    for part, sp, gr in zip(c["parts"], seg_prm, sgr):
        ss, m, o = part["ss"], part["m"], part["off"]
        dC = dH[g0:g0 + m]
        if ss.levels == 2:
            gr["b_c2"] += dC.sum(0)
            gr["W_c2"] += dC.T @ part["Y"].reshape(m, ss.k2 * d)
            dY = (dC @ _f64(sp["W_c2"])).reshape(m, ss.k2, d)
        else:
            dY = dC.reshape(m, 1, d)
        gr["b_c1"] += dY.sum((0, 1))
        groups = part["Xb"].reshape(m, ss.k2, ss.k1 * d)
        gr["W_c1"] += dY.reshape(m * ss.k2, d).T @ groups.reshape(m * ss.k2, ss.k1 * d)
        dgroups = dY @ _f64(sp["W_c1"])
        dX[o:o + ss.L] += unpartition(dgroups.reshape(m, ss.P, d), ss, ss.L)
        g0 += m
    return dX, sgr, grads


def partition_w(A, spec):
    """``partition`` for a per-token array of any width (2D patches)."""
    p, gh, gw = spec.patch, spec.grid_h, spec.grid_w
    w = A.shape[1]
    g = A.reshape(gh // p, p, gw // p, p, w)
    return g.transpose(0, 2, 1, 3, 4).reshape(-1, p * p, w)


def layer_bwd(spec, prm, X, G, H_in=None, t=None, dH_out=None, caches=None):
    """Backward of ``layer_fwd`` (chain rule through Eqs. partition ...
    inj-*).  Returns (dX [B, L, d], dH_in [B, m, d], grads{name: array}).
    ``caches`` may pass the activations a ``layer_fwd(..., return_cache=True)``
    of the same inputs returned, instead of recomputing them."""
    X = _f64(X)
    G = _f64(G)
    if caches is None:
        _, _, caches = layer_fwd(spec, prm, X, H_in, t, return_cache=True)
    grads = {k: np.zeros(np.shape(v)) for k, v in prm.items()
             if k.startswith(("W_", "b_", "w_"))}
    dXs, dHs = [], []
    for b in range(X.shape[0]):
        dho = None if dH_out is None else _f64(dH_out[b])
        dX, dH_in = _bwd_one(spec, prm, X[b], caches[b], G[b], dho, grads)
        dXs.append(dX)
        dHs.append(dH_in)
    return np.stack(dXs), np.stack(dHs), grads
