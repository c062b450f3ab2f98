"""A stack of causal 1D ProxyFormer layers with per-layer ratios (Sec. 3.6).

Layer l's proxy state H is carried into layer l+1 only when both use the same
P; otherwise the next layer re-extracts its proxies from the local stream
(H_in = NULL).  The backward walks the layers in reverse with the matching
rule for dH.  All arithmetic happens in the library (ProxyLayer calls).
"""
from __future__ import annotations

from typing import Dict, List, Optional

import torch

from .layer import ProxyLayer


class ProxyStack:
    def __init__(self, specs: List, params: List[Dict], device="cuda"):
        assert len(specs) == len(params) and specs
        self.specs = specs
        from . import layer_desc, proxy_layer_workspace_size
        need = max(max(proxy_layer_workspace_size(layer_desc(s), f) for f in (0, 1))
                   for s in specs)
        self.ws = torch.empty(max(need, 16), dtype=torch.uint8, device=device)
        self.layers = [ProxyLayer(s, p, device, ws=self.ws) for s, p in zip(specs, params)]
        s0 = specs[0]
        width = getattr(s0, "d_fine", 0) or s0.d  # token width
        self.X = [torch.empty((s0.batch, s0.L, width), dtype=torch.bfloat16, device=device)
                  for _ in range(len(specs) + 1)]
        self.H = [lay.empty_proxy() for lay in self.layers]
        self.dX = [torch.empty_like(self.X[0]) for _ in range(2)]
        self.dH = [lay.empty_proxy() for lay in self.layers]

    def carries(self, l: int) -> bool:
        """True if layer l receives H from layer l-1 (same block size)."""
        return l > 0 and self.specs[l].P == self.specs[l - 1].P

    def forward(self, X0: torch.Tensor, train: bool = True) -> torch.Tensor:
        self.X[0].copy_(X0)
        for l, lay in enumerate(self.layers):
            H_in = self.H[l - 1] if self.carries(l) else None
            lay.forward(self.X[l], H_in, X_out=self.X[l + 1], H_out=self.H[l], train=train)
        return self.X[-1]

    def prefill(self, X_hist: torch.Tensor, caches: List) -> torch.Tensor:
        """Prefill stage (Sec. 3.8): each layer's inference forward over the
        history, which also fills that layer's proxy KV cache (a ProxyKVCache
        whose proxy key/value projection is the layer's own W_k, W_v) with the
        keys and values its proxy attention computed.  Returns the last
        layer's output."""
        assert len(caches) == len(self.layers)
        self.X[0].copy_(X_hist)
        for l, (lay, cache) in enumerate(zip(self.layers, caches)):
            H_in = self.H[l - 1] if self.carries(l) else None
            lay.prefill(self.X[l], cache, H_in, X_out=self.X[l + 1], H_out=self.H[l])
        return self.X[-1]

    def backward(self, G: torch.Tensor) -> torch.Tensor:
        n = len(self.layers)
        dX_out = G
        for l in reversed(range(n)):
            lay = self.layers[l]
            H_in = self.H[l - 1] if self.carries(l) else None
            dH_out = self.dH[l + 1] if l + 1 < n and self.carries(l + 1) else None
            dX = self.dX[l % 2]
            lay.backward(self.X[l], dX_out, H_in, dH_out=dH_out, dX=dX,
                         dH_in=self.dH[l] if self.carries(l) else None)
            dX_out = dX
        return dX_out
