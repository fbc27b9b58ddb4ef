"""GB300 (sm_103a) pruned-pool batched-decode MoE layer of SlimWise (arXiv 2609.34117).

The layer runs as hand-written CUDA kernels in ``libslimwise.so`` behind the C
ABI of ``include/slimwise_moe.h``; ``binding`` is the thin ctypes layer with the
same function names.  Importing this package does not load the library; the
first call does, and raises if it has not been built (``build.build()``).
"""
from .binding import (  # noqa: F401
    SlimwiseError,
    alloc_workspace,
    load,
    slimwise_moe_compact_layer,
    slimwise_moe_decode,
    slimwise_moe_decode_ex,
    slimwise_moe_decode_full,
    slimwise_moe_decode_shared,
    slimwise_moe_device_status,
    slimwise_moe_expert_stats,
    slimwise_moe_group,
    slimwise_moe_route,
    slimwise_moe_select_retained,
    slimwise_moe_shared_workspace_size,
    slimwise_moe_workspace_size,
)
