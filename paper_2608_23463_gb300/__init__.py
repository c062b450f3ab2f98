"""Python binding of libproxyformer.so, the sm_103a ProxyFormer hot path.

Argument marshalling only: every step of the layer, append and decode runs in
the library's CUDA kernels.  The functions below carry the C ABI's names
(``include/proxyformer.h``) and take device pointers as ints, or tensors (their
``data_ptr()`` is passed), or None for NULL.  A non-OK status raises
``ProxyFormerError``.  There is no fallback: if the library is not built the
first call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Any, Dict, Optional

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libproxyformer.so")

PF_OK, PF_ERR_INVALID_ARG, PF_ERR_UNSUPPORTED, PF_ERR_WORKSPACE = 0, 1, 2, 3
PF_ERR_CAPACITY, PF_ERR_CUDA, PF_ERR_TIMEOUT = 4, 5, 6
PF_CAUSAL_1D, PF_BIDIR_1D, PF_BIDIR_2D = 0, 1, 2
PF_INJ_ADD, PF_INJ_GATED, PF_INJ_AFFINE, PF_INJ_CROSS = 0, 1, 2, 3
PF_F32, PF_BF16 = 0, 1
PF_F_ATTENTION, PF_F_IDENTITY, PF_F_MLP = 0, 1, 2

_c_i32 = ctypes.c_int32
_vp = ctypes.c_void_p


class ProxyFormerError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"pf_status {status}: {message}")
        self.status = status


class LayerDesc(ctypes.Structure):
    _fields_ = [(n, _c_i32) for n in ("batch", "L", "grid_h", "grid_w", "patch", "d", "n_heads",
                                      "P", "levels", "k1", "k2", "mode", "inject", "dtype",
                                      "d_fine", "interact", "rope")]


_PARAM_NAMES = ("W_c1", "b_c1", "W_c2", "b_c2", "W_qkv", "W_o", "W_d2", "b_d2", "W_d1", "b_d1",
                "w_x", "w_dlt", "b_g", "W_t1", "b_t1", "W_t2", "b_t2", "W_qa", "b_a", "W_kvx",
                "W_ox", "W_m1", "b_m1", "W_m2", "b_m2")


class LayerParams(ctypes.Structure):
    _fields_ = [(n, _vp) for n in _PARAM_NAMES]


class LayerGrads(ctypes.Structure):
    _fields_ = [(n, _vp) for n in _PARAM_NAMES]


class Segment(ctypes.Structure):
    _fields_ = [(n, _c_i32) for n in ("L", "P", "k1", "k2")]


_SEG_NAMES = ("W_c1", "b_c1", "W_c2", "b_c2", "W_d1", "b_d1", "W_d2", "b_d2")


class SegmentParams(ctypes.Structure):
    _fields_ = [(n, _vp) for n in _SEG_NAMES]


class DecodeDesc(ctypes.Structure):
    _fields_ = [(n, _c_i32) for n in ("batch", "d", "n_heads", "P", "levels", "k1", "k2",
                                      "capacity")]


class KVCache(ctypes.Structure):
    _fields_ = [("K_proxy", _vp), ("V_proxy", _vp), ("X_open", _vp), ("K_open", _vp),
                ("V_open", _vp), ("n_proxy", _vp), ("n_open", _vp)]


class DecodeParams(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("W_qkv", "W_o", "rms_w", "W_a1", "b_a1", "W_a2", "b_a2")]


class AppendParams(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("W_c1", "b_c1", "W_c2", "b_c2", "W_kvh")]


EXPORTED = ("proxy_layer_check", "proxy_layer_saved_size", "proxy_layer_workspace_size",
            "proxy_layer_fwd", "proxy_layer_bwd", "proxy_decode_workspace_size",
            "proxy_decode_step", "proxy_append_workspace_size", "proxy_kv_append",
            "proxy_prefill_workspace_size", "proxy_kv_prefill", "proxy_layer_prefill",
            "proxy_segments_saved_size", "proxy_segments_workspace_size", "proxy_segments_fwd",
            "proxy_segments_bwd",
            "pf_last_error", "pf_sync_check", "pf_gemm_bf16", "pf_timing_enable",
            "pf_timing_collect", "pf_timing_label", "pf_timing_ms", "pf_timing_launches",
            "pf_timing_flops", "pf_timing_bytes", "proxy_layer_bwd_noalloc",
            "pf_debug_set_wait_limit_ns", "pf_debug_gemm_skip_loads", "pf_probe_ffma")

_lib: Optional[ctypes.CDLL] = None


def load(path: str = LIB_PATH) -> ctypes.CDLL:
    """Load (once) and type the shared library; raises if it is not built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ProxyFormerError(PF_ERR_CUDA, f"{path} is not built; run "
                               "`python -m paper_2608_23463_gb300.buildlib`")
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER
    sz = ctypes.c_size_t
    lib.proxy_layer_check.argtypes = [P(LayerDesc)]
    lib.proxy_layer_check.restype = ctypes.c_int
    lib.proxy_layer_saved_size.argtypes = [P(LayerDesc)]
    lib.proxy_layer_saved_size.restype = sz
    lib.proxy_layer_workspace_size.argtypes = [P(LayerDesc), ctypes.c_int]
    lib.proxy_layer_workspace_size.restype = sz
    lib.proxy_layer_fwd.argtypes = [P(LayerDesc), P(LayerParams), _vp, _vp, _vp, _vp, _vp, _vp,
                                    _vp, sz, _vp]
    lib.proxy_layer_fwd.restype = ctypes.c_int
    lib.proxy_layer_bwd.argtypes = [P(LayerDesc), P(LayerParams), _vp, _vp, _vp, _vp, _vp, _vp,
                                    _vp, _vp, P(LayerGrads), _vp, sz, _vp]
    lib.proxy_layer_bwd.restype = ctypes.c_int
    lib.proxy_decode_workspace_size.argtypes = [P(DecodeDesc)]
    lib.proxy_decode_workspace_size.restype = sz
    lib.proxy_decode_step.argtypes = [P(DecodeDesc), P(DecodeParams), _vp, P(KVCache), _vp, _vp,
                                      sz, _vp]
    lib.proxy_decode_step.restype = ctypes.c_int
    lib.proxy_append_workspace_size.argtypes = [P(DecodeDesc)]
    lib.proxy_append_workspace_size.restype = sz
    lib.proxy_kv_append.argtypes = [P(DecodeDesc), P(AppendParams), _vp, P(KVCache), _vp, sz, _vp]
    lib.proxy_kv_append.restype = ctypes.c_int
    lib.proxy_prefill_workspace_size.argtypes = [P(DecodeDesc), ctypes.c_int32]
    lib.proxy_prefill_workspace_size.restype = sz
    lib.proxy_kv_prefill.argtypes = [P(DecodeDesc), P(AppendParams), P(DecodeParams), _vp,
                                     ctypes.c_int32, _vp, P(KVCache), _vp, sz, _vp]
    lib.proxy_kv_prefill.restype = ctypes.c_int
    lib.proxy_layer_prefill.argtypes = [P(LayerDesc), P(LayerParams), P(DecodeDesc),
                                        P(DecodeParams), _vp, _vp, _vp, _vp, P(KVCache), _vp, sz,
                                        _vp]
    lib.proxy_layer_prefill.restype = ctypes.c_int
    lib.proxy_segments_saved_size.argtypes = [P(LayerDesc), ctypes.c_int32, P(Segment)]
    lib.proxy_segments_saved_size.restype = sz
    lib.proxy_segments_workspace_size.argtypes = [P(LayerDesc), ctypes.c_int32, P(Segment),
                                                  ctypes.c_int]
    lib.proxy_segments_workspace_size.restype = sz
    lib.proxy_segments_fwd.argtypes = [P(LayerDesc), ctypes.c_int32, P(Segment), P(LayerParams),
                                       P(SegmentParams), _vp, _vp, _vp, _vp, sz, _vp]
    lib.proxy_segments_fwd.restype = ctypes.c_int
    lib.proxy_segments_bwd.argtypes = [P(LayerDesc), ctypes.c_int32, P(Segment), P(LayerParams),
                                       P(SegmentParams), _vp, _vp, _vp, _vp, P(LayerGrads),
                                       P(SegmentParams), _vp, sz, _vp]
    lib.proxy_segments_bwd.restype = ctypes.c_int
    lib.pf_last_error.argtypes = []
    lib.pf_last_error.restype = ctypes.c_char_p
    lib.pf_sync_check.argtypes = [_vp]
    lib.pf_sync_check.restype = ctypes.c_int
    lib.pf_gemm_bf16.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_int, _vp, ctypes.c_int, _vp,
                                 ctypes.c_int, _vp, ctypes.c_int, _vp]
    lib.pf_gemm_bf16.restype = ctypes.c_int
    lib.pf_timing_enable.argtypes = [ctypes.c_int]
    lib.pf_timing_enable.restype = None
    lib.pf_timing_collect.argtypes = []
    lib.pf_timing_collect.restype = ctypes.c_int
    lib.pf_timing_label.argtypes = [ctypes.c_int]
    lib.pf_timing_label.restype = ctypes.c_char_p
    for n in ("pf_timing_ms", "pf_timing_flops", "pf_timing_bytes"):
        getattr(lib, n).argtypes = [ctypes.c_int]
        getattr(lib, n).restype = ctypes.c_double
    lib.proxy_layer_bwd_noalloc.argtypes = [P(LayerDesc), P(LayerParams), _vp, _vp, _vp, _vp, _vp,
                                            _vp, _vp, _vp, P(LayerGrads), _vp]
    lib.proxy_layer_bwd_noalloc.restype = ctypes.c_int
    lib.pf_timing_launches.argtypes = [ctypes.c_int]
    lib.pf_timing_launches.restype = ctypes.c_int
    lib.pf_debug_set_wait_limit_ns.argtypes = [ctypes.c_ulonglong]
    lib.pf_debug_set_wait_limit_ns.restype = ctypes.c_int
    lib.pf_debug_gemm_skip_loads.argtypes = [ctypes.c_int]
    lib.pf_debug_gemm_skip_loads.restype = ctypes.c_int
    lib.pf_probe_ffma.argtypes = [_vp, ctypes.c_int, ctypes.c_int, _vp]
    lib.pf_probe_ffma.restype = ctypes.c_int
    _lib = lib
    return lib


def _ptr(x: Any) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def _check(status: int) -> None:
    if status != PF_OK:
        msg = load().pf_last_error()
        raise ProxyFormerError(status, msg.decode() if msg else "")


def layer_desc(spec) -> LayerDesc:
    """LayerDesc from any object with the descriptor's attribute names."""
    return LayerDesc(*(int(getattr(spec, f, 0) or 0) for f, _ in LayerDesc._fields_))


def layer_params(tensors: Dict[str, Any], grads: bool = False):
    cls = LayerGrads if grads else LayerParams
    return cls(*(_ptr(tensors.get(n)) for n in _PARAM_NAMES))


def proxy_layer_check(desc: LayerDesc) -> int:
    return load().proxy_layer_check(ctypes.byref(desc))


def proxy_layer_saved_size(desc: LayerDesc) -> int:
    return load().proxy_layer_saved_size(ctypes.byref(desc))


def proxy_layer_workspace_size(desc: LayerDesc, for_backward: int) -> int:
    return load().proxy_layer_workspace_size(ctypes.byref(desc), int(for_backward))


def proxy_layer_fwd(desc, params, X, H_in, t, X_out, H_out, saved, ws, ws_bytes, stream=None):
    _check(load().proxy_layer_fwd(ctypes.byref(desc), ctypes.byref(params), _ptr(X), _ptr(H_in),
                                  _ptr(t), _ptr(X_out), _ptr(H_out), _ptr(saved), _ptr(ws),
                                  int(ws_bytes), stream))


def proxy_layer_bwd(desc, params, X, H_in, t, saved, dX_out, dH_out, dX, dH_in, grads, ws,
                    ws_bytes, stream=None):
    _check(load().proxy_layer_bwd(ctypes.byref(desc), ctypes.byref(params), _ptr(X), _ptr(H_in),
                                  _ptr(t), _ptr(saved), _ptr(dX_out), _ptr(dH_out), _ptr(dX),
                                  _ptr(dH_in), ctypes.byref(grads), _ptr(ws), int(ws_bytes),
                                  stream))


def proxy_layer_bwd_noalloc(desc, params, X, H_in, t, saved, dX_out, dH_out, dX, dH_in, grads,
                            stream=None):
    """proxy_layer_bwd for callers that cannot provide a workspace: scratch comes
    from a fixed device array inside the library (PF_NOALLOC_SCRATCH_BYTES)."""
    _check(load().proxy_layer_bwd_noalloc(ctypes.byref(desc), ctypes.byref(params), _ptr(X),
                                          _ptr(H_in), _ptr(t), _ptr(saved), _ptr(dX_out),
                                          _ptr(dH_out), _ptr(dX), _ptr(dH_in), ctypes.byref(grads),
                                          stream))


PF_NOALLOC_SCRATCH_BYTES = 16 << 20


def proxy_decode_workspace_size(desc: DecodeDesc) -> int:
    return load().proxy_decode_workspace_size(ctypes.byref(desc))


def proxy_decode_step(desc, params, x, cache, y, ws, ws_bytes, stream=None):
    _check(load().proxy_decode_step(ctypes.byref(desc), ctypes.byref(params), _ptr(x),
                                    ctypes.byref(cache), _ptr(y), _ptr(ws), int(ws_bytes), stream))


def proxy_append_workspace_size(desc: DecodeDesc) -> int:
    return load().proxy_append_workspace_size(ctypes.byref(desc))


def proxy_kv_append(desc, params, H_in, cache, ws, ws_bytes, stream=None):
    _check(load().proxy_kv_append(ctypes.byref(desc), ctypes.byref(params), _ptr(H_in),
                                  ctypes.byref(cache), _ptr(ws), int(ws_bytes), stream))


def proxy_prefill_workspace_size(desc: DecodeDesc, L_hist: int) -> int:
    return load().proxy_prefill_workspace_size(ctypes.byref(desc), int(L_hist))


def proxy_kv_prefill(desc, aparams, dparams, X_hist, L_hist, H_in, cache, ws, ws_bytes,
                     stream=None):
    _check(load().proxy_kv_prefill(ctypes.byref(desc), ctypes.byref(aparams),
                                   ctypes.byref(dparams), _ptr(X_hist), int(L_hist), _ptr(H_in),
                                   ctypes.byref(cache), _ptr(ws), int(ws_bytes), stream))


def proxy_layer_prefill(desc, params, cdesc, dparams, X, H_in, X_out, H_out, cache, ws,
                        ws_bytes, stream=None):
    _check(load().proxy_layer_prefill(ctypes.byref(desc), ctypes.byref(params),
                                      ctypes.byref(cdesc), ctypes.byref(dparams), _ptr(X),
                                      _ptr(H_in), _ptr(X_out), _ptr(H_out), ctypes.byref(cache),
                                      _ptr(ws), int(ws_bytes), stream))


def segment_array(specs) -> "ctypes.Array":
    """pf_segment array from (L, P[, k1, k2]) tuples."""
    arr = (Segment * len(specs))()
    for a, sp in zip(arr, specs):
        a.L, a.P = int(sp[0]), int(sp[1])
        a.k1, a.k2 = (int(sp[2]), int(sp[3])) if len(sp) > 2 else (0, 0)
    return arr


def segment_params(tensors_list) -> "ctypes.Array":
    """pf_segment_params (or pf_segment_grads, same layout) array."""
    arr = (SegmentParams * len(tensors_list))()
    for a, t in zip(arr, tensors_list):
        for n in _SEG_NAMES:
            setattr(a, n, _ptr(t.get(n)))
    return arr


def proxy_segments_saved_size(desc, segs) -> int:
    return load().proxy_segments_saved_size(ctypes.byref(desc), len(segs), segs)


def proxy_segments_workspace_size(desc, segs, for_backward: int) -> int:
    return load().proxy_segments_workspace_size(ctypes.byref(desc), len(segs), segs,
                                                int(for_backward))


def proxy_segments_fwd(desc, segs, shared, seg_params, X, X_out, saved, ws, ws_bytes,
                       stream=None):
    _check(load().proxy_segments_fwd(ctypes.byref(desc), len(segs), segs, ctypes.byref(shared),
                                     seg_params, _ptr(X), _ptr(X_out), _ptr(saved), _ptr(ws),
                                     int(ws_bytes), stream))


def proxy_segments_bwd(desc, segs, shared, seg_params, X, saved, dX_out, dX, grads, seg_grads,
                       ws, ws_bytes, stream=None):
    _check(load().proxy_segments_bwd(ctypes.byref(desc), len(segs), segs, ctypes.byref(shared),
                                     seg_params, _ptr(X), _ptr(saved), _ptr(dX_out), _ptr(dX),
                                     ctypes.byref(grads), seg_grads, _ptr(ws), int(ws_bytes),
                                     stream))


def pf_sync_check(stream=None) -> None:
    _check(load().pf_sync_check(stream))


def pf_last_error() -> str:
    msg = load().pf_last_error()
    return msg.decode() if msg else ""


def pf_gemm_bf16(M, N, K, A, a_mn, B, b_mn, D, ldd, stream=None):
    _check(load().pf_gemm_bf16(int(M), int(N), int(K), _ptr(A), int(a_mn), _ptr(B), int(b_mn),
                               _ptr(D), int(ldd), stream))


def pf_debug_set_wait_limit_ns(ns: int) -> None:
    """Time limit of every bounded wait in the library's kernels (0: default)."""
    _check(load().pf_debug_set_wait_limit_ns(int(ns)))


def pf_debug_gemm_skip_loads(on: bool) -> None:
    """Test hook: the GEMM kernel issues no operand loads while on."""
    _check(load().pf_debug_gemm_skip_loads(1 if on else 0))


def pf_probe_ffma(out, blocks: int, iters: int, stream=None) -> None:
    """Launch the fp32 FMA peak probe (2 * blocks * 512 * 8 * iters FLOPs)."""
    _check(load().pf_probe_ffma(_ptr(out), int(blocks), int(iters), stream))


def pf_timing_enable(on: bool) -> None:
    load().pf_timing_enable(1 if on else 0)


def pf_timing_collect():
    """Per-label launch timing since pf_timing_enable (caller has synchronised):
    {label: dict(ms=total, launches=n, flops=per launch, bytes=per launch)}."""
    lib = load()
    out = {}
    for i in range(lib.pf_timing_collect()):
        out[lib.pf_timing_label(i).decode()] = dict(
            ms=lib.pf_timing_ms(i), launches=lib.pf_timing_launches(i),
            flops=lib.pf_timing_flops(i), bytes=lib.pf_timing_bytes(i))
    return out


def build(verbose: bool = False) -> str:
    from .buildlib import build as _build
    return _build(verbose=verbose)
