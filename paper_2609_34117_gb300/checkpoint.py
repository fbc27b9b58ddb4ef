"""Compact (pruned) checkpoint of one MoE layer.

SlimWise serves decode from a pool K' of m' retained experts (Sec. 3.1).
Restricting the router to K' with the Eq. 2 mask is the same as loading a
pruned checkpoint that holds only the retained experts' weights and router
rows; a PD-disaggregated decode instance keeps only that compact form.  It is
built once, offline, from the full layer by the library's compaction kernels
(slimwise_moe_compact_layer): rows of the retained experts in ascending id.
Either form then runs on the CUDA decode path:

    masked:  slimwise_moe_decode(x, router_w, retained_idx, ...)   on [E, ...]
    compact: slimwise_moe_decode_full(x, router_c, ...)            on [m', ...]

The two give identical outputs, and compact expert j is original expert
`ids[j]` in the selections.
"""
from __future__ import annotations

import torch

from . import binding


def compact_layer(w_gate_up: torch.Tensor, w_down: torch.Tensor, router_w: torch.Tensor,
                  retained_idx: torch.Tensor, stream=None):
    """Return (w_gate_up_c, w_down_c, router_w_c, ids): the retained experts'
    weights [m', 2I, H], [m', H, I] and router rows [m', H], and the sorted
    original ids (int32, on the device) they came from.  Synchronises the
    stream to check the ids; raises ValueError on repeated or out-of-range ids."""
    ret = retained_idx.to(device=w_gate_up.device, dtype=torch.int32).flatten().contiguous()
    if ret.numel() == 0:
        raise ValueError("retained ids must be in [0, E)")
    gu_c, d_c, wr_c, ids = binding.slimwise_moe_compact_layer(w_gate_up, w_down, router_w, ret,
                                                              stream=stream)
    if int(ids[0].item()) < 0:
        raise ValueError("retained ids must be distinct and in [0, E)")
    return gu_c, d_c, wr_c, ids
