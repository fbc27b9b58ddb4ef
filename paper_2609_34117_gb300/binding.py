"""Thin ctypes binding of libslimwise.so (include/slimwise_moe.h).

Argument marshalling only: every step of the layer runs in the library's CUDA
kernels.  PyTorch tensors supply device memory and the current stream.  The
functions keep the C names; each returns the output tensors it was given or
allocated and raises SlimwiseError on a non-zero status.  There is no CPU
path: without the built library every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lock = threading.Lock()
_lib = None

SLIMWISE_OK = 0
STATUS_NAMES = {0: "ok", 1: "invalid argument", 2: "unsupported shape or alignment",
                3: "workspace too small", 4: "CUDA error", 5: "device-side error"}
DEVERR_PIPELINE_TIMEOUT = 0x1
DEVERR_DEPENDENCY_TIMEOUT = 0x2
DEVERR_DUPLICATE_RETAINED = 0x4
DEVERR_BAD_RETAINED = 0x8
DEVERR_BAD_TOPK = 0x10
DEVERR_TMEM_PAIR = 0x20

EXPORTED = (
    "slimwise_status_string", "slimwise_moe_workspace_size", "slimwise_moe_decode",
    "slimwise_moe_decode_full", "slimwise_moe_decode_ex", "slimwise_moe_route",
    "slimwise_moe_group", "slimwise_moe_device_status", "slimwise_moe_decode_noalloc",
    "slimwise_moe_shared_workspace_size", "slimwise_moe_decode_shared",
    "slimwise_moe_decode_shared_ex", "slimwise_moe_expert_stats", "slimwise_moe_select_retained",
    "slimwise_moe_noalloc_device_status", "slimwise_moe_compact_layer",
)


class SlimwiseError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {STATUS_NAMES.get(status, 'unknown')} (status {status})")
        self.status = status


class Shape(ctypes.Structure):
    _fields_ = [("num_tokens", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("num_experts", ctypes.c_int32), ("inter", ctypes.c_int32)]


class DecodeOpts(ctypes.Structure):
    _fields_ = [("ffn_begin", ctypes.c_void_p), ("ffn_end", ctypes.c_void_p),
                ("disable_pdl", ctypes.c_int32), ("grid_ctas", ctypes.c_int32),
                ("wait_limit_ns", ctypes.c_int64), ("test_starve_first_down", ctypes.c_int32),
                ("ffn_items", ctypes.c_int32)]


def library_path() -> str:
    """The library this process loads: $SLIMWISE_LIBRARY if set (e.g. the
    timeline-stamping build, build.TRACE_LIB_PATH), else the in-tree build."""
    return os.environ.get("SLIMWISE_LIBRARY") or _build.LIB_PATH


def load(path: str | None = None) -> ctypes.CDLL:
    """Load libslimwise.so (or `path`, or $SLIMWISE_LIBRARY); raises if it has
    not been built."""
    global _lib
    with _lock:
        if _lib is None:
            p = path or library_path()
            if not os.path.exists(p):
                raise RuntimeError(f"libslimwise.so not built ({p}); run paper_2609_34117_gb300.build.build()")
            lib = ctypes.CDLL(p)
            P, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
            SP = ctypes.POINTER(Shape)
            lib.slimwise_status_string.argtypes = [ctypes.c_int]
            lib.slimwise_status_string.restype = ctypes.c_char_p
            lib.slimwise_moe_workspace_size.argtypes = [SP, i32, ctypes.POINTER(sz)]
            lib.slimwise_moe_decode.argtypes = [P, P, P, i32, P, P, i32, P, P, SP, P, sz]
            lib.slimwise_moe_decode_full.argtypes = [P, P, P, P, i32, P, P, SP, P, sz]
            lib.slimwise_moe_decode_ex.argtypes = [P, P, P, i32, P, P, i32, P, P, SP, P, sz,
                                                   ctypes.POINTER(DecodeOpts)]
            lib.slimwise_moe_route.argtypes = [P, P, P, i32, i32, P, SP, P, sz] + [P] * 8
            lib.slimwise_moe_group.argtypes = [P, i32, P, SP, P, sz] + [P] * 6
            lib.slimwise_moe_device_status.argtypes = [P, P, ctypes.POINTER(i32)]
            lib.slimwise_moe_decode_noalloc.argtypes = [P, P, P, i32, P, P, i32, P, P, SP]
            lib.slimwise_moe_noalloc_device_status.argtypes = [P, ctypes.POINTER(i32)]
            lib.slimwise_moe_shared_workspace_size.argtypes = [SP, i32, i32, ctypes.POINTER(sz)]
            lib.slimwise_moe_decode_shared.argtypes = [P, P, P, i32, P, P, i32, P, P, P, i32,
                                                       P, P, SP, P, sz]
            lib.slimwise_moe_decode_shared_ex.argtypes = [P, P, P, i32, P, P, i32, P, P, P, i32,
                                                          P, P, SP, P, sz,
                                                          ctypes.POINTER(DecodeOpts)]
            lib.slimwise_moe_expert_stats.argtypes = [P, P, P, P, i32, P, P, P, SP, P, sz]
            lib.slimwise_moe_select_retained.argtypes = [P, i32, i32, i32, P, P]
            lib.slimwise_moe_compact_layer.argtypes = [P, P, P, P, i32, SP, P, P, P, P, P]
            for name in EXPORTED[1:]:
                getattr(lib, name).restype = ctypes.c_int
            _lib = lib
    return _lib


def _check(rc: int, what: str):
    if rc != SLIMWISE_OK:
        raise SlimwiseError(rc, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, dtype, name):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _shape_of(hidden, w_gate_up, num_tokens=None):
    E, two_i, H = w_gate_up.shape
    B = hidden.shape[0] if num_tokens is None else num_tokens
    return Shape(int(B), int(H), int(E), int(two_i // 2))


def slimwise_moe_workspace_size(num_tokens: int, hidden: int, num_experts: int, inter: int,
                                top_k: int) -> int:
    out = ctypes.c_size_t(0)
    s = Shape(num_tokens, hidden, num_experts, inter)
    _check(load().slimwise_moe_workspace_size(ctypes.byref(s), top_k, ctypes.byref(out)),
           "slimwise_moe_workspace_size")
    return int(out.value)


def alloc_workspace(num_tokens, hidden, num_experts, inter, top_k, device=None) -> torch.Tensor:
    n = slimwise_moe_workspace_size(num_tokens, hidden, num_experts, inter, top_k)
    return torch.empty(n, dtype=torch.uint8, device=device or "cuda")


def _prep(hidden, router_w, w_gate_up, w_down, top_k, out, workspace):
    _dev(hidden, torch.bfloat16, "hidden")
    _dev(router_w, torch.float32, "router_w")
    _dev(w_gate_up, torch.bfloat16, "w_gate_up")
    _dev(w_down, torch.bfloat16, "w_down")
    s = _shape_of(hidden, w_gate_up)
    if out is None:
        out = torch.empty((s.num_tokens, s.hidden), dtype=torch.bfloat16, device=hidden.device)
    _dev(out, torch.bfloat16, "out")
    if workspace is None:
        workspace = alloc_workspace(s.num_tokens, s.hidden, s.num_experts, s.inter, top_k,
                                    hidden.device)
    return s, out, workspace


def slimwise_moe_shared_workspace_size(num_tokens: int, hidden: int, num_experts: int, inter: int,
                                       top_k: int, inter_shared: int) -> int:
    out = ctypes.c_size_t(0)
    s = Shape(num_tokens, hidden, num_experts, inter)
    _check(load().slimwise_moe_shared_workspace_size(ctypes.byref(s), top_k, int(inter_shared),
                                                     ctypes.byref(out)),
           "slimwise_moe_shared_workspace_size")
    return int(out.value)


def slimwise_moe_decode_shared(hidden, router_w, retained_idx, w_gate_up, w_down, top_k,
                               w_shared_gate, w_shared_gate_up, w_shared_down, out=None,
                               workspace=None, stream=None, ffn_events=None, disable_pdl=False,
                               grid_ctas=0):
    """Decode MoE layer with a shared expert under a sigmoid gate (Sec. 3.3);
    retained_idx None = full pool.  Launch options as slimwise_moe_decode_ex.
    Returns `out`."""
    _dev(hidden, torch.bfloat16, "hidden")
    _dev(router_w, torch.float32, "router_w")
    _dev(w_gate_up, torch.bfloat16, "w_gate_up")
    _dev(w_down, torch.bfloat16, "w_down")
    _dev(w_shared_gate, torch.float32, "w_shared_gate")
    _dev(w_shared_gate_up, torch.bfloat16, "w_shared_gate_up")
    _dev(w_shared_down, torch.bfloat16, "w_shared_down")
    s = _shape_of(hidden, w_gate_up)
    inter_shared = int(w_shared_gate_up.shape[0]) // 2
    if out is None:
        out = torch.empty((s.num_tokens, s.hidden), dtype=torch.bfloat16, device=hidden.device)
    _dev(out, torch.bfloat16, "out")
    if workspace is None:
        n = slimwise_moe_shared_workspace_size(s.num_tokens, s.hidden, s.num_experts, s.inter,
                                               top_k, inter_shared)
        workspace = torch.empty(n, dtype=torch.uint8, device=hidden.device)
    n_ret = 0
    if retained_idx is not None:
        _dev(retained_idx, torch.int32, "retained_idx")
        n_ret = int(retained_idx.numel())
    args = (_ptr(hidden), _ptr(router_w), _ptr(retained_idx), n_ret, _ptr(w_gate_up), _ptr(w_down),
            int(top_k), _ptr(w_shared_gate), _ptr(w_shared_gate_up), _ptr(w_shared_down),
            inter_shared, _ptr(out), _stream(stream), ctypes.byref(s), _ptr(workspace),
            workspace.numel())
    if ffn_events is None and not disable_pdl and not grid_ctas:
        _check(load().slimwise_moe_decode_shared(*args), "slimwise_moe_decode_shared")
    else:
        opts = _opts(ffn_events, disable_pdl, grid_ctas)
        _check(load().slimwise_moe_decode_shared_ex(*args, ctypes.byref(opts)),
               "slimwise_moe_decode_shared_ex")
    return out


def slimwise_moe_decode(hidden, router_w, retained_idx, w_gate_up, w_down, top_k,
                        out=None, workspace=None, stream=None):
    """Decode MoE layer over the retained pool (Sec. 3.1, Eq. 2); returns `out`."""
    s, out, workspace = _prep(hidden, router_w, w_gate_up, w_down, top_k, out, workspace)
    _dev(retained_idx, torch.int32, "retained_idx")
    _check(load().slimwise_moe_decode(
        _ptr(hidden), _ptr(router_w), _ptr(retained_idx), int(retained_idx.numel()),
        _ptr(w_gate_up), _ptr(w_down), int(top_k), _ptr(out), _stream(stream),
        ctypes.byref(s), _ptr(workspace), workspace.numel()), "slimwise_moe_decode")
    return out


def slimwise_moe_decode_full(hidden, router_w, w_gate_up, w_down, top_k, out=None,
                             workspace=None, stream=None):
    """Decode MoE layer over the full pool; returns `out`."""
    s, out, workspace = _prep(hidden, router_w, w_gate_up, w_down, top_k, out, workspace)
    _check(load().slimwise_moe_decode_full(
        _ptr(hidden), _ptr(router_w), _ptr(w_gate_up), _ptr(w_down), int(top_k), _ptr(out),
        _stream(stream), ctypes.byref(s), _ptr(workspace), workspace.numel()),
        "slimwise_moe_decode_full")
    return out


CRITERIA = {"mass": 0, "ean": 1, "reap": 2}


def slimwise_moe_expert_stats(hidden, router_w, w_gate_up, w_down, top_k, stats=None, out=None,
                              workspace=None, stream=None):
    """One calibration batch of importance statistics (Sec. 2.3), full pool.
    `stats` (fp64 [E, 4], device) accumulates; returns (stats, layer output)."""
    s, out, workspace = _prep(hidden, router_w, w_gate_up, w_down, top_k, out, workspace)
    if stats is None:
        stats = torch.zeros((s.num_experts, 4), dtype=torch.float64, device=hidden.device)
    _dev(stats, torch.float64, "stats")
    _check(load().slimwise_moe_expert_stats(
        _ptr(hidden), _ptr(router_w), _ptr(w_gate_up), _ptr(w_down), int(top_k), _ptr(stats),
        _ptr(out), _stream(stream), ctypes.byref(s), _ptr(workspace), workspace.numel()),
        "slimwise_moe_expert_stats")
    return stats, out


def slimwise_moe_select_retained(stats, n_retained, criterion="reap", stream=None):
    """Retained set from statistics: int32 [n_retained] device ids, ascending."""
    _dev(stats, torch.float64, "stats")
    ids = torch.empty(int(n_retained), dtype=torch.int32, device=stats.device)
    _check(load().slimwise_moe_select_retained(_ptr(stats), int(stats.shape[0]), int(n_retained),
                                               CRITERIA[criterion], _ptr(ids), _stream(stream)),
           "slimwise_moe_select_retained")
    return ids


def slimwise_moe_compact_layer(w_gate_up, w_down, router_w, retained_idx, stream=None):
    """Compact checkpoint of the retained experts (Sec. 3.1), built by the
    library's kernels: returns (w_gate_up_c [m', 2I, H], w_down_c [m', H, I],
    router_w_c [m', H], ids_c int32 [m']) with the experts in ascending original
    id.  Asynchronous on the stream: on a repeated or out-of-range id every
    ids_c entry is -1 and the other outputs are left unwritten."""
    _dev(w_gate_up, torch.bfloat16, "w_gate_up")
    _dev(w_down, torch.bfloat16, "w_down")
    _dev(router_w, torch.float32, "router_w")
    _dev(retained_idx, torch.int32, "retained_idx")
    E, two_i, H = (int(v) for v in w_gate_up.shape)
    m = int(retained_idx.numel())
    s = Shape(0, H, E, two_i // 2)
    dev = w_gate_up.device
    gu_c = torch.empty((m, two_i, H), dtype=torch.bfloat16, device=dev)
    d_c = torch.empty((m,) + tuple(w_down.shape[1:]), dtype=torch.bfloat16, device=dev)
    wr_c = torch.empty((m, H), dtype=torch.float32, device=dev)
    ids_c = torch.empty(m, dtype=torch.int32, device=dev)
    _check(load().slimwise_moe_compact_layer(_ptr(w_gate_up), _ptr(w_down), _ptr(router_w),
                                             _ptr(retained_idx), m, ctypes.byref(s), _ptr(gu_c),
                                             _ptr(d_c), _ptr(wr_c), _ptr(ids_c), _stream(stream)),
           "slimwise_moe_compact_layer")
    return gu_c, d_c, wr_c, ids_c


def _opts(ffn_events, disable_pdl, grid_ctas, wait_limit_ns=0, test_starve_first_down=False,
          ffn_items=0):
    opts = DecodeOpts(None, None, int(bool(disable_pdl)), int(grid_ctas), int(wait_limit_ns),
                      int(bool(test_starve_first_down)), int(ffn_items))
    if ffn_events is not None:
        opts.ffn_begin = ctypes.c_void_p(ffn_events[0].cuda_event)
        opts.ffn_end = ctypes.c_void_p(ffn_events[1].cuda_event)
    return opts


def slimwise_moe_decode_ex(hidden, router_w, retained_idx, w_gate_up, w_down, top_k,
                           out=None, workspace=None, stream=None, ffn_events=None,
                           disable_pdl=False, grid_ctas=0, wait_limit_ns=0,
                           test_starve_first_down=False, ffn_items=0):
    """slimwise_moe_decode with launch options; retained_idx None = full pool.

    ffn_events: optional (begin, end) torch.cuda.Event pair recorded around the
    expert-FFN kernel on the launch stream.  wait_limit_ns: limit of the FFN
    kernel's bounded waits (0: 1 s).  test_starve_first_down: tests only, makes
    the first down item's dependency wait run out.  ffn_items: form of the FFN
    work items (0 or -1 the default, 1 CTA-pair items where the layer allows).
    """
    s, out, workspace = _prep(hidden, router_w, w_gate_up, w_down, top_k, out, workspace)
    if retained_idx is not None:
        _dev(retained_idx, torch.int32, "retained_idx")
    opts = _opts(ffn_events, disable_pdl, grid_ctas, wait_limit_ns, test_starve_first_down,
                 ffn_items)
    n_ret = 0 if retained_idx is None else int(retained_idx.numel())
    _check(load().slimwise_moe_decode_ex(
        _ptr(hidden), _ptr(router_w), _ptr(retained_idx), n_ret, _ptr(w_gate_up), _ptr(w_down),
        int(top_k), _ptr(out), _stream(stream), ctypes.byref(s), _ptr(workspace),
        workspace.numel(), ctypes.byref(opts)), "slimwise_moe_decode_ex")
    return out


def _group_outputs(B, k, E, device):
    i32 = dict(dtype=torch.int32, device=device)
    return {"counts": torch.empty(E, **i32), "offsets": torch.empty(E + 1, **i32),
            "union_ids": torch.empty(E, **i32), "union_size": torch.empty(1, **i32),
            "perm": torch.empty(B * k, **i32), "pos": torch.empty(B * k, **i32)}


def slimwise_moe_route(hidden, router_w, retained_idx, top_k, num_experts, inter=64,
                       workspace=None, stream=None):
    """Routing + grouping only; returns a dict of device tensors."""
    _dev(hidden, torch.bfloat16, "hidden")
    _dev(router_w, torch.float32, "router_w")
    B, H = hidden.shape
    s = Shape(B, H, num_experts, inter)
    if workspace is None:
        workspace = alloc_workspace(B, H, num_experts, inter, top_k, hidden.device)
    if retained_idx is not None:
        _dev(retained_idx, torch.int32, "retained_idx")
    res = {"topk_idx": torch.empty((B, top_k), dtype=torch.int32, device=hidden.device),
           "topk_gate": torch.empty((B, top_k), dtype=torch.float32, device=hidden.device)}
    res.update(_group_outputs(B, top_k, num_experts, hidden.device))
    n_ret = 0 if retained_idx is None else int(retained_idx.numel())
    _check(load().slimwise_moe_route(
        _ptr(hidden), _ptr(router_w), _ptr(retained_idx), n_ret, int(top_k), _stream(stream),
        ctypes.byref(s), _ptr(workspace), workspace.numel(),
        *[_ptr(res[n]) for n in ("topk_idx", "topk_gate", "counts", "offsets", "union_ids",
                                  "union_size", "perm", "pos")]), "slimwise_moe_route")
    return res


def slimwise_moe_group(topk_idx, num_experts, hidden=128, inter=64, workspace=None, stream=None):
    """Grouping of given selections int32 [B, k]; returns a dict of device tensors."""
    _dev(topk_idx, torch.int32, "topk_idx")
    B, k = topk_idx.shape
    s = Shape(B, hidden, num_experts, inter)
    if workspace is None:
        workspace = alloc_workspace(B, hidden, num_experts, inter, k, topk_idx.device)
    res = _group_outputs(B, k, num_experts, topk_idx.device)
    _check(load().slimwise_moe_group(
        _ptr(topk_idx), int(k), _stream(stream), ctypes.byref(s), _ptr(workspace),
        workspace.numel(), *[_ptr(res[n]) for n in ("counts", "offsets", "union_ids",
                                                      "union_size", "perm", "pos")]),
        "slimwise_moe_group")
    return res


def slimwise_moe_device_status(workspace, stream=None) -> int:
    """Device error bits of the last call on `workspace` (synchronises the stream)."""
    flags = ctypes.c_int32(0)
    rc = load().slimwise_moe_device_status(_ptr(workspace), _stream(stream), ctypes.byref(flags))
    if rc not in (0, 5):
        _check(rc, "slimwise_moe_device_status")
    return int(flags.value)


def slimwise_moe_decode_noalloc(hidden, router_w, retained_idx, w_gate_up, w_down, top_k,
                                out, stream=None):
    """The decode layer for callers that cannot allocate device memory.

    The library keeps this entry point's scratch in a fixed 16 MiB device
    array, so the call needs no workspace; `out` (bf16 [B, H]) must be given.
    retained_idx None = full pool.  Calls that may overlap on the GPU race on
    the shared array.
    """
    _dev(hidden, torch.bfloat16, "hidden")
    _dev(router_w, torch.float32, "router_w")
    _dev(w_gate_up, torch.bfloat16, "w_gate_up")
    _dev(w_down, torch.bfloat16, "w_down")
    _dev(out, torch.bfloat16, "out")
    if retained_idx is not None:
        _dev(retained_idx, torch.int32, "retained_idx")
    s = _shape_of(hidden, w_gate_up)
    n_ret = 0 if retained_idx is None else int(retained_idx.numel())
    _check(load().slimwise_moe_decode_noalloc(
        _ptr(hidden), _ptr(router_w), _ptr(retained_idx), n_ret, _ptr(w_gate_up), _ptr(w_down),
        int(top_k), _ptr(out), _stream(stream), ctypes.byref(s)), "slimwise_moe_decode_noalloc")
    return out


def slimwise_moe_noalloc_device_status(stream=None) -> int:
    """Device error bits of the last slimwise_moe_decode_noalloc call on the
    current device (synchronises the stream)."""
    flags = ctypes.c_int32(0)
    rc = load().slimwise_moe_noalloc_device_status(_stream(stream), ctypes.byref(flags))
    if rc not in (0, 5):
        _check(rc, "slimwise_moe_noalloc_device_status")
    return int(flags.value)
