"""Compact (pruned) checkpoint of one MoE layer.

SlimWise serves decode from a pool K' of m' retained experts (Sec. 3.1).
Restricting the router to K' with the Eq. 2 mask is the same as loading a
pruned checkpoint that holds only the retained experts' weights and router
rows; a PD-disaggregated decode instance keeps only that compact form.  This
module builds it once, offline, from the full layer: rows of the retained
experts in ascending id order.  It is model preparation, not a decode step --
the decode path runs in the CUDA library, on either form:

    masked:  slimwise_moe_decode(x, router_w, retained_idx, ...)   on [E, ...]
    compact: slimwise_moe_decode_full(x, router_c, ...)            on [m', ...]

The two give identical outputs, and compact expert j is original expert
`ids[j]` in the selections.
"""
from __future__ import annotations

import torch


def compact_layer(w_gate_up: torch.Tensor, w_down: torch.Tensor, router_w: torch.Tensor,
                  retained_idx: torch.Tensor):
    """Return (w_gate_up_c, w_down_c, router_w_c, ids): the retained experts'
    weights [m', 2I, H], [m', H, I] and router rows [m', H], and the sorted
    original ids (int32) they came from.  Raises on repeated or out-of-range ids."""
    E = w_gate_up.shape[0]
    ids = torch.sort(retained_idx.to(torch.int64).flatten()).values
    if ids.numel() == 0 or int(ids[0]) < 0 or int(ids[-1]) >= E:
        raise ValueError("retained ids must be in [0, E)")
    if ids.numel() > 1 and bool((ids[1:] == ids[:-1]).any()):
        raise ValueError("retained ids must be distinct")
    sel = ids.to(w_gate_up.device)
    return (w_gate_up.index_select(0, sel).contiguous(),
            w_down.index_select(0, sel.to(w_down.device)).contiguous(),
            router_w.index_select(0, sel.to(router_w.device)).contiguous(),
            ids.to(torch.int32))
