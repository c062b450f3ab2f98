"""Seeded synthetic inputs for the ProxyFormer layer, append and decode paths.

This module is the only code shared by the CUDA path's tests/bench and the CPU
oracle.  It draws random numbers and lays them out in the shapes of the layer's
tensors; it holds none of the method's arithmetic (no compression, attention,
decompression or injection).

Conventions fixed here (the layer's parameter shapes, ProxyFormer Sec. 3):
  * every weight matrix is stored [out, in] (row-major): y = W @ x + b;
  * flattening a block of tokens is token-major: vec index p*d + ch;
  * level 1 of a two-level cascade is the token side (k1 tokens -> 1 row),
    level 2 the proxy side (k2 rows -> 1 proxy), P = k1*k2 (Eq. factor);
  * decompression mirrors it: level 2 maps a proxy to k2 rows, level 1 maps
    each row to k1 tokens (Eq. factor-dec).

Random draws use numpy's PCG64 (``numpy.random.default_rng(seed)``) in the fill
order given by ``layer_param_shapes`` followed by the activations.  Matrices are
Xavier-uniform U(+-sqrt(6/(fan_in+fan_out))); bias and gate vectors U(+-0.1);
norm weights 1 + U(+-0.1).  For bf16 workloads every value is rounded once to
the nearest bf16 (ties to even) so both sides of a comparison start from the
same representable numbers.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Dict, Optional

import numpy as np

# mode / inject / dtype codes; they mirror the C header's enums.
CAUSAL_1D, BIDIR_1D, BIDIR_2D = 0, 1, 2
F_ATTENTION, F_IDENTITY, F_MLP = 0, 1, 2  # proxy interaction
INJ_ADD, INJ_GATED, INJ_AFFINE, INJ_CROSS = 0, 1, 2, 3
F32, BF16 = 0, 1

TEMB_DIM = 256  # width of the sinusoidal timestep embedding (2D layer)


@dataclasses.dataclass(frozen=True)
class LayerSpec:
    """Shape of one ProxyFormer layer (Alg. 1) plus its variant flags."""

    batch: int
    L: int
    d: int
    n_heads: int
    P: int
    levels: int = 1
    k1: int = 0
    k2: int = 0
    mode: int = CAUSAL_1D
    inject: int = INJ_GATED
    dtype: int = BF16
    grid_h: int = 0
    grid_w: int = 0
    patch: int = 0
    d_fine: int = 0  # token width when it differs from the proxy width d
    interact: int = F_ATTENTION
    rope: int = 0  # rotate the proxies' queries and keys (attention only)

    def __post_init__(self):
        if self.levels == 1:
            object.__setattr__(self, "k1", self.P)
            object.__setattr__(self, "k2", 1)

    @property
    def df(self) -> int:
        """Token (local stream) width: d_fine, else d."""
        return self.d_fine or self.d

    @property
    def m(self) -> int:
        """Number of blocks (proxies) per sequence, m = ceil(L/P)."""
        return -(-self.L // self.P)

    @property
    def dh(self) -> int:
        return self.d // self.n_heads


@dataclasses.dataclass(frozen=True)
class DecodeSpec:
    """Shape of the proxy KV-cache decode state (Sec. 3.7/3.8)."""

    batch: int
    d: int
    n_heads: int
    P: int
    levels: int = 1
    k1: int = 0
    k2: int = 0
    capacity: int = 0

    def __post_init__(self):
        if self.levels == 1:
            object.__setattr__(self, "k1", self.P)
            object.__setattr__(self, "k2", 1)

    @property
    def dh(self) -> int:
        return self.d // self.n_heads


def default_factors(P: int):
    """k1 = 2**ceil(log2(P)/2), k2 = P/k1 (16->4x4, 64->8x8, 128->16x8)."""
    k1 = 1 << math.ceil(math.log2(P) / 2)
    return k1, P // k1


def round_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16, ties to even (no NaN input)."""
    a = np.array(a, dtype=np.float32, copy=True)
    u = a.view(np.uint32)  # finite inputs: the sum below cannot wrap
    u += np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    u &= np.uint32(0xFFFF0000)
    return a


def _finish(a: np.ndarray, dtype: int) -> np.ndarray:
    a = a.astype(np.float32)
    return round_bf16(a) if dtype == BF16 else a


def layer_param_shapes(spec: LayerSpec) -> Dict[str, tuple]:
    """Parameter names and shapes, in generator fill order."""
    d, P, k1, k2, df = spec.d, spec.P, spec.k1, spec.k2, spec.df
    s = {}
    s["W_c1"] = (d, k1 * df)
    s["b_c1"] = (d,)
    if spec.levels == 2:
        s["W_c2"] = (d, k2 * d)
        s["b_c2"] = (d,)
    if spec.interact == F_ATTENTION:
        s["W_qkv"] = (3 * d, d)
        s["W_o"] = (d, d)
    elif spec.interact == F_MLP:
        s["W_m1"] = (4 * d, d)
        s["b_m1"] = (4 * d,)
        s["W_m2"] = (d, 4 * d)
        s["b_m2"] = (d,)
    if spec.inject == INJ_CROSS:
        # token queries stacked over the per-head gate rows; proxy keys and
        # values of the injection; its output projection
        s["W_qa"] = (d + spec.n_heads, d)
        s["b_a"] = (spec.n_heads,)
        s["W_kvx"] = (2 * d, d)
        s["W_ox"] = (d, d)
        return s
    out_tok = 2 * d if spec.inject == INJ_AFFINE else df
    if spec.levels == 2:
        s["W_d2"] = (k2 * d, d)
        s["b_d2"] = (k2 * d,)
    s["W_d1"] = (k1 * out_tok, d)
    s["b_d1"] = (k1 * out_tok,)
    if spec.inject == INJ_GATED:
        s["w_x"] = (df,)
        s["w_dlt"] = (df,)
        s["b_g"] = (df,)
    if spec.mode == BIDIR_2D:
        s["W_t1"] = (d, TEMB_DIM)
        s["b_t1"] = (d,)
        s["W_t2"] = (2 * d, d)
        s["b_t2"] = (2 * d,)
    return s


def _xavier(rng, shape):
    fan_out, fan_in = shape
    bound = math.sqrt(6.0 / (fan_in + fan_out))
    return rng.uniform(-bound, bound, size=shape)


def make_layer_params(spec: LayerSpec, seed: int) -> Dict[str, np.ndarray]:
    rng = np.random.default_rng(seed)
    out = {}
    for name, shape in layer_param_shapes(spec).items():
        if name in ("W_qkv", "W_kvx"):  # d x d matrices drawn one after another
            d = spec.d
            a = np.concatenate([_xavier(rng, (d, d)) for _ in range(shape[0] // d)], axis=0)
        elif len(shape) == 2:
            a = _xavier(rng, shape)
        else:
            a = rng.uniform(-0.1, 0.1, size=shape)
        out[name] = _finish(a, spec.dtype)
    return out


def make_layer_inputs(spec: LayerSpec, seed: int, with_h_in: bool = False,
                      with_grads: bool = True) -> Dict[str, np.ndarray]:
    """Params + activations.  X ~ N(0,1) [B, L, d]; G (upstream grad of X_out)
    ~ N(0,1); dH_out ~ N(0,1); H_in ~ N(0,1) if requested; t ~ U(0,1) [B]."""
    p = make_layer_params(spec, seed)
    rng = np.random.default_rng(seed + 0x5EED)
    B, L, d, m, df = spec.batch, spec.L, spec.d, spec.m, spec.df
    p["X"] = _finish(rng.standard_normal((B, L, df), dtype=np.float32), spec.dtype)
    if with_h_in:
        p["H_in"] = rng.standard_normal((B, m, d), dtype=np.float32)
    if spec.mode == BIDIR_2D:
        p["t"] = rng.uniform(0.0, 1.0, size=(B,)).astype(np.float32)
    if with_grads:
        p["G"] = _finish(rng.standard_normal((B, L, df), dtype=np.float32), spec.dtype)
        p["dH_out"] = rng.standard_normal((B, m, d), dtype=np.float32)
    return p


def decode_param_shapes(spec: DecodeSpec) -> Dict[str, tuple]:
    d, k1, k2, nh = spec.d, spec.k1, spec.k2, spec.n_heads
    s = {"W_qkv": (3 * d, d), "W_o": (d, d), "rms_w": (d,),
         "W_a1": (d // 8, d), "b_a1": (d // 8,), "W_a2": (nh, d // 8), "b_a2": (nh,),
         "W_c1": (d, k1 * d), "b_c1": (d,)}
    if spec.levels == 2:
        s["W_c2"] = (d, k2 * d)
        s["b_c2"] = (d,)
    s["W_kvh"] = (2 * d, d)
    return s


def make_decode_params(spec: DecodeSpec, seed: int) -> Dict[str, np.ndarray]:
    rng = np.random.default_rng(seed)
    out = {}
    for name, shape in decode_param_shapes(spec).items():
        if name in ("W_qkv", "W_kvh"):
            d = spec.d
            nmat = shape[0] // d
            a = np.concatenate([_xavier(rng, (d, d)) for _ in range(nmat)], axis=0)
        elif len(shape) == 2:
            a = _xavier(rng, shape)
        elif name == "rms_w":
            a = 1.0 + rng.uniform(-0.1, 0.1, size=shape)
        else:
            a = rng.uniform(-0.1, 0.1, size=shape)
        out[name] = round_bf16(a.astype(np.float32))
    return out


def decode_spec_for_layer(spec: "LayerSpec", capacity: int) -> DecodeSpec:
    """The proxy KV cache of one causal layer: its width, heads and block
    factors, room for `capacity` proxies per sequence."""
    return DecodeSpec(batch=spec.batch, d=spec.d, n_heads=spec.n_heads, P=spec.P,
                      levels=spec.levels, k1=spec.k1 if spec.levels == 2 else 0,
                      k2=spec.k2 if spec.levels == 2 else 0, capacity=capacity)


def decode_params_for_layer(spec: "LayerSpec", layer_params: Dict[str, np.ndarray],
                            seed: int) -> Dict[str, np.ndarray]:
    """Decode-side parameters of a layer: the layer's own compression weights
    (W_c1, b_c1, W_c2, b_c2) and, as the proxy key/value projection W_kvh, the
    key and value rows of the layer's W_qkv; the decode-only weights (token
    W_qkv, W_o, RMSNorm, gate MLP) drawn from `seed`."""
    out = make_decode_params(decode_spec_for_layer(spec, 1), seed)
    for k in ("W_c1", "b_c1", "W_c2", "b_c2"):
        if k in layer_params:
            out[k] = layer_params[k]
    out["W_kvh"] = np.ascontiguousarray(layer_params["W_qkv"][spec.d:])
    return out


def make_decode_state(spec: DecodeSpec, seed: int, n_proxy, n_open):
    """Cache contents ~ N(0,1): K/V proxy rows [B, capacity, d] (rows past
    n_proxy[b] are filled too, and must be ignored), open-block features and
    their K/V [B, P, d] (slots past n_open[b] likewise), new token x [B, d]."""
    rng = np.random.default_rng(seed + 0xDEC)
    B, d, P, cap = spec.batch, spec.d, spec.P, spec.capacity
    st = {}
    st["K_proxy"] = round_bf16(rng.standard_normal((B, cap, d), dtype=np.float32))
    st["V_proxy"] = round_bf16(rng.standard_normal((B, cap, d), dtype=np.float32))
    st["X_open"] = round_bf16(rng.standard_normal((B, P, d), dtype=np.float32))
    st["K_open"] = round_bf16(rng.standard_normal((B, P, d), dtype=np.float32))
    st["V_open"] = round_bf16(rng.standard_normal((B, P, d), dtype=np.float32))
    st["x"] = round_bf16(rng.standard_normal((B, d), dtype=np.float32))
    st["n_proxy"] = np.asarray(n_proxy, dtype=np.int32).reshape(B)
    st["n_open"] = np.asarray(n_open, dtype=np.int32).reshape(B)
    return st


# Workloads used by the tests and the bench (the paper's layer shapes).
def spec_c1():
    """1D causal layer, fwd, fp32: L=4096, d=256, 4x64 heads, P=64 single-level."""
    return LayerSpec(batch=1, L=4096, d=256, n_heads=4, P=64, dtype=F32)


def spec_c2():
    """1D causal layer, fwd+bwd, bf16: L=65536, d=1024, 16x64 heads, P=64."""
    return LayerSpec(batch=1, L=65536, d=1024, n_heads=16, P=64)


def spec_c3_layer(P: int = 64):
    """One layer of the 12-layer stack: L=262144, d=1024, 16x64, factorised."""
    k1, k2 = default_factors(P)
    return LayerSpec(batch=1, L=262144, d=1024, n_heads=16, P=P, levels=2, k1=k1, k2=k2)


def spec_cross_layer():
    """The causal headline layer with gated cross-attention injection:
    L=262144, d=1024, 16x64 heads, P=64 as 8x8."""
    return LayerSpec(batch=1, L=262144, d=1024, n_heads=16, P=64, levels=2, k1=8, k2=8,
                     inject=INJ_CROSS)


def spec_lm_history():
    """The language model's history layer (Sec. 3.3, Sec. 5.1): 64-wide
    tokens compressed into 512-wide proxies, 8x64 heads, P = 64, a
    1048576-token history."""
    return LayerSpec(batch=1, L=1048576, d=512, n_heads=8, P=64, d_fine=64)


SEGMENT_KEYS = ("W_c1", "b_c1", "W_c2", "b_c2", "W_d1", "b_d1", "W_d2", "b_d2")


def make_segment_params(d: int, n_heads: int, levels: int, segs, seed: int):
    """Parameters of a layer with temporal-distance ratios: the shared ones
    (proxy attention and gate: W_qkv, W_o, w_x, w_dlt, b_g) and one set of
    compression / decompression weights per segment (L, P[, k1, k2])."""
    shared, per = None, []
    for i, sg in enumerate(segs):
        kw = dict(k1=sg[2], k2=sg[3]) if levels == 2 else {}
        sp = LayerSpec(batch=1, L=sg[0], d=d, n_heads=n_heads, P=sg[1], levels=levels, **kw)
        p = make_layer_params(sp, seed + i)
        per.append({k: v for k, v in p.items() if k in SEGMENT_KEYS})
        if shared is None:
            shared = {k: v for k, v in p.items() if k not in SEGMENT_KEYS}
    return shared, per


C3_RATIOS = (16, 16, 32, 32, 64, 64, 64, 64, 128, 128, 256, 256)


def spec_c4():
    """Proxy-only KV decode: B=8, d=2048, 16x128 heads, P=64, 16384 cached proxies."""
    return DecodeSpec(batch=8, d=2048, n_heads=16, P=64, capacity=16384)


def spec_c5():
    """2D bidirectional layer: B=4, 512x512 grid, d=512, 8x64 heads, 8x8 patches."""
    return LayerSpec(batch=4, L=512 * 512, d=512, n_heads=8, P=64, mode=BIDIR_2D,
                     inject=INJ_AFFINE, grid_h=512, grid_w=512, patch=8)
