"""A causal layer whose blocks grow coarser with temporal distance (Sec. 3.6).

``ProxySegmentLayer`` keeps the shared parameters (proxy attention, gate),
each segment's compression / decompression parameters, their gradients and
the saved activations on the device and calls ``proxy_segments_fwd`` /
``proxy_segments_bwd``.  It does no arithmetic of its own.
"""
from __future__ import annotations

from typing import Dict, List, Sequence

import numpy as np
import torch

from . import (layer_desc, layer_params, proxy_segments_bwd, proxy_segments_fwd,
               proxy_segments_saved_size, proxy_segments_workspace_size, segment_array,
               segment_params)


def _dev(a, device):
    return torch.from_numpy(np.ascontiguousarray(a)).to(
        device=device, dtype=torch.bfloat16 if np.ndim(a) == 2 else torch.float32)


class ProxySegmentLayer:
    def __init__(self, spec, segs: Sequence[tuple], shared: Dict[str, np.ndarray],
                 seg_params: List[Dict[str, np.ndarray]], device="cuda"):
        self.spec, self.device = spec, device
        self.desc = layer_desc(spec)
        self.segs = segment_array(segs)
        self.p = {k: _dev(v, device) for k, v in shared.items()}
        self.sp = [{k: _dev(v, device) for k, v in d.items()} for d in seg_params]
        self.p_struct = layer_params(self.p)
        self.sp_struct = segment_params(self.sp)
        f32 = lambda t: torch.zeros(t.shape, dtype=torch.float32, device=device)
        self.grads = {k: f32(v) for k, v in self.p.items()}
        self.seg_grads = [{k: f32(v) for k, v in d.items()} for d in self.sp]
        self.g_struct = layer_params(self.grads, grads=True)
        self.sg_struct = segment_params(self.seg_grads)
        self.saved = torch.empty(max(proxy_segments_saved_size(self.desc, self.segs), 16),
                                 dtype=torch.uint8, device=device)
        need = max(proxy_segments_workspace_size(self.desc, self.segs, f) for f in (0, 1))
        self.ws = torch.empty(max(need, 16), dtype=torch.uint8, device=device)

    def forward(self, X: torch.Tensor, X_out: torch.Tensor = None) -> torch.Tensor:
        X_out = torch.empty_like(X) if X_out is None else X_out
        proxy_segments_fwd(self.desc, self.segs, self.p_struct, self.sp_struct, X, X_out,
                           self.saved, self.ws, self.ws.numel(),
                           torch.cuda.current_stream().cuda_stream)
        return X_out

    def backward(self, X: torch.Tensor, G: torch.Tensor, dX: torch.Tensor = None) -> torch.Tensor:
        dX = torch.empty_like(X) if dX is None else dX
        proxy_segments_bwd(self.desc, self.segs, self.p_struct, self.sp_struct, X, self.saved, G,
                           dX, self.g_struct, self.sg_struct, self.ws, self.ws.numel(),
                           torch.cuda.current_stream().cuda_stream)
        return dX
