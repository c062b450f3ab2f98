"""CPU oracle for the ProxyFormer layer, KV append and decode step.

TEST INFRASTRUCTURE ONLY.  Nothing in the product path may import this package:
only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s ``cpu_baseline``
/ ``--impl reference`` legs use it.  It is a plain, slow, float64 restatement of
the paper's equations, sharing no code with the CUDA library.

Parity status per function (what pins it, see ``tests/test_oracle_pins.py``):
  * partition / compression / cascade ........ pinned (factorisation identity,
    conv2d identity, P=1 reduction, block-index probe)
  * proxy attention (causal, bidirectional) ... pinned (torch SDPA, brute force,
    one-hot mask probe, causality perturbation)
  * decompression / routing / injection ........ pinned (P=1 reduction, gate
    limits reduce to Eq. inj-add / identity, causality, LayerNorm vs torch)
  * backward (all variants) .................... pinned by central finite
    differences of the forward in float64
  * decode step / KV append .................... pinned (torch SDPA for both
    attentions, alpha gate limits, streaming consistency with the layer's
    compression)
  * timestep embedding constants of the 2D layer (frequencies, the 1000 scale)
    and the width of the alpha MLP: parity unpinned -- they are this library's
    own definitions; only finite differences and self-consistency check them.
"""
from .layer import layer_fwd, layer_bwd, timestep_embedding  # noqa: F401
from .decode import decode_step, kv_append, compress_block  # noqa: F401
