"""Device-resident proxy KV cache and decode/append calls (PyTorch holds memory).

``ProxyKVCache`` keeps the decode-side parameters, the cache state and the
workspaces on the device and calls ``proxy_decode_step`` / ``proxy_kv_append``
/ ``proxy_kv_prefill`` on the current CUDA stream.  It does no arithmetic of
its own.
"""
from __future__ import annotations

from typing import Dict

import numpy as np
import torch

from . import (AppendParams, DecodeDesc, DecodeParams, KVCache, _ptr, proxy_append_workspace_size,
               proxy_decode_step, proxy_decode_workspace_size, proxy_kv_append, proxy_kv_prefill,
               proxy_prefill_workspace_size)


def _dev(a, dtype, device):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device=device, dtype=dtype)


class ProxyKVCache:
    """Proxy-only KV cache of one layer (Sec. 3.8) plus its decode parameters."""

    def __init__(self, spec, params: Dict[str, np.ndarray], state: Dict[str, np.ndarray],
                 device="cuda"):
        self.spec = spec
        self.desc = DecodeDesc(spec.batch, spec.d, spec.n_heads, spec.P, spec.levels, spec.k1,
                               spec.k2, spec.capacity)
        bf, f32 = torch.bfloat16, torch.float32
        self.p = {k: _dev(v, bf if np.ndim(v) == 2 else f32, device) for k, v in params.items()}
        self.s = {k: _dev(state[k], bf, device)
                  for k in ("K_proxy", "V_proxy", "X_open", "K_open", "V_open")}
        self.s["n_proxy"] = _dev(state["n_proxy"], torch.int32, device)
        self.s["n_open"] = _dev(state["n_open"], torch.int32, device)
        g = lambda k: _ptr(self.p.get(k))
        self.dp = DecodeParams(g("W_qkv"), g("W_o"), g("rms_w"), g("W_a1"), g("b_a1"), g("W_a2"),
                               g("b_a2"))
        self.ap = AppendParams(g("W_c1"), g("b_c1"), g("W_c2"), g("b_c2"), g("W_kvh"))
        c = self.s
        self.cache = KVCache(_ptr(c["K_proxy"]), _ptr(c["V_proxy"]), _ptr(c["X_open"]),
                             _ptr(c["K_open"]), _ptr(c["V_open"]), _ptr(c["n_proxy"]),
                             _ptr(c["n_open"]))
        nd = proxy_decode_workspace_size(self.desc)
        na = proxy_append_workspace_size(self.desc)
        self.ws = torch.empty(max(nd, na, 16), dtype=torch.uint8, device=device)

    def step(self, x: torch.Tensor, y: torch.Tensor = None) -> torch.Tensor:
        y = torch.empty_like(x) if y is None else y
        proxy_decode_step(self.desc, self.dp, x, self.cache, y, self.ws, self.ws.numel(),
                          torch.cuda.current_stream().cuda_stream)
        return y

    def capture_step(self, x: torch.Tensor, y: torch.Tensor) -> "torch.cuda.CUDAGraph":
        """Record one decode step on fixed x / y buffers as a CUDA graph.

        Capturing only records the launches; each ``replay()`` then runs one step
        (the open-block counters live on the device, so consecutive replays fill
        consecutive slots).  Per-launch timing must be off while capturing."""
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            self.step(x, y)
        return g

    def append(self, H_in: torch.Tensor = None) -> None:
        proxy_kv_append(self.desc, self.ap, H_in, self.cache, self.ws, self.ws.numel(),
                        torch.cuda.current_stream().cuda_stream)

    def prefill(self, X_hist: torch.Tensor, H_in: torch.Tensor = None,
                ws: torch.Tensor = None) -> None:
        """Fill the cache from a history X_hist [batch, L_hist, d] (bf16): its
        complete blocks' proxies and the remaining tokens' open block.  ``ws``
        may hold a workspace of proxy_prefill_workspace_size bytes (allocated
        here if None)."""
        L_hist = int(X_hist.shape[1])
        need = proxy_prefill_workspace_size(self.desc, L_hist)
        if ws is None or ws.numel() < need:
            ws = torch.empty(max(need, 16), dtype=torch.uint8, device=X_hist.device)
        proxy_kv_prefill(self.desc, self.ap, self.dp, X_hist, L_hist, H_in, self.cache, ws,
                         ws.numel(), torch.cuda.current_stream().cuda_stream)
