"""Device-resident ProxyFormer layer around the C ABI (PyTorch holds memory).

``ProxyLayer`` keeps one layer's parameters, gradients, saved tensors and
workspaces in device memory and calls ``proxy_layer_fwd`` / ``proxy_layer_bwd``
on the current CUDA stream.  It does no arithmetic of its own.
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np
import torch

from . import (PF_BF16, layer_desc, layer_params, proxy_layer_bwd, proxy_layer_fwd,
               proxy_layer_prefill, proxy_layer_saved_size, proxy_layer_workspace_size)


def _stream() -> int:
    return torch.cuda.current_stream().cuda_stream


def to_device(a: np.ndarray, dtype: torch.dtype, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device=device,
                                                                        dtype=dtype)


class ProxyLayer:
    """One layer (Alg. 1) with device buffers sized from the descriptor."""

    def __init__(self, spec, params: Dict[str, np.ndarray], device="cuda",
                 ws: Optional[torch.Tensor] = None):
        self.spec = spec
        self.desc = layer_desc(spec)
        self.act_dtype = torch.bfloat16 if spec.dtype == PF_BF16 else torch.float32
        self.device = device
        self.params: Dict[str, torch.Tensor] = {}
        for k, v in params.items():
            if not k.startswith(("W_", "b_", "w_")):
                continue
            dt = self.act_dtype if np.ndim(v) == 2 else torch.float32
            self.params[k] = to_device(v, dt, device)
        self.p_struct = layer_params(self.params)
        self.grads = {k: torch.zeros(v.shape, dtype=torch.float32, device=device)
                      for k, v in self.params.items()}
        self.g_struct = layer_params(self.grads, grads=True)
        self.saved = torch.empty(max(proxy_layer_saved_size(self.desc), 16), dtype=torch.uint8,
                                 device=device)
        self.ws_fwd_bytes = proxy_layer_workspace_size(self.desc, 0)
        self.ws_bwd_bytes = proxy_layer_workspace_size(self.desc, 1)
        need = max(self.ws_fwd_bytes, self.ws_bwd_bytes, 16)
        if ws is not None and ws.numel() >= need:
            self.ws = ws  # shared with other layers that run on the same stream
        else:
            self.ws = torch.empty(need, dtype=torch.uint8, device=device)

    def empty_act(self) -> torch.Tensor:
        s = self.spec
        width = getattr(s, "d_fine", 0) or s.d  # token width
        return torch.empty((s.batch, s.L, width), dtype=self.act_dtype, device=self.device)

    def empty_proxy(self) -> torch.Tensor:
        s = self.spec
        return torch.empty((s.batch, s.m, s.d), dtype=torch.float32, device=self.device)

    def forward(self, X, H_in=None, t=None, X_out=None, H_out=None, train=True):
        X_out = self.empty_act() if X_out is None else X_out
        proxy_layer_fwd(self.desc, self.p_struct, X, H_in, t, X_out, H_out,
                        self.saved if train else None, self.ws, self.ws.numel(), _stream())
        return X_out

    def prefill(self, X, cache, H_in=None, X_out=None, H_out=None):
        """Inference forward over a history plus the fill of `cache` (a
        ProxyKVCache of this layer) from the forward's own proxy keys and
        values (Sec. 3.8); see proxy_layer_prefill."""
        X_out = self.empty_act() if X_out is None else X_out
        proxy_layer_prefill(self.desc, self.p_struct, cache.desc, cache.dp, X, H_in, X_out, H_out,
                            cache.cache, self.ws, self.ws.numel(), _stream())
        return X_out

    def backward(self, X, dX_out, H_in=None, t=None, dH_out=None, dX=None, dH_in=None):
        dX = self.empty_act() if dX is None else dX
        proxy_layer_bwd(self.desc, self.p_struct, X, H_in, t, self.saved, dX_out, dH_out, dX,
                        dH_in, self.g_struct, self.ws, self.ws.numel(), _stream())
        return dX
