"""C-ABI checks that need no GPU: the library loads, exports every symbol the
header declares, sizes its workspace, and rejects bad arguments on the host
before touching CUDA."""
import ctypes
import os
import re

import pytest

from paper_2609_34117_gb300 import binding, build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return binding.load()


def _declared_functions():
    with open(os.path.join(ROOT, "include", "slimwise_moe.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?(?:int|char\s*\*|const char\s*\*)\s*\*?\s*(slimwise_\w+)\s*\(",
                                 text, re.M)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert len(names) >= 8, names
    for n in names:
        assert hasattr(lib, n), n
    assert set(binding.EXPORTED) == set(names)


def test_status_strings(lib):
    for code, name in binding.STATUS_NAMES.items():
        assert lib.slimwise_status_string(code).decode() == name


def _ws(B, H, E, I, k):
    return binding.slimwise_moe_workspace_size(B, H, E, I, k)


def test_workspace_size_grows_with_batch_and_covers_buffers(lib):
    H, E, I, k = 2048, 128, 768, 8
    prev = 0
    for B in (1, 8, 64, 256, 512):
        n = _ws(B, H, E, I, k)
        # grouped hidden rows, activations and expert outputs (all bf16)
        assert n >= B * k * (2 * H + 2 * I + 2 * H)
        assert n > prev
        prev = n
    assert _ws(0, H, E, I, k) > 0


@pytest.mark.parametrize("B,H,E,I,k,code", [
    (4, 100, 16, 128, 2, 2),     # H not a multiple of 128
    (4, 32896, 16, 128, 2, 2),   # H above 32768
    (4, 256, 16, 96, 2, 2),      # I not a multiple of 64
    (4, 256, 2000, 128, 2, 2),   # too many experts
    (4, 256, 16, 128, 0, 1),     # top_k = 0
    (4, 256, 16, 128, 33, 1),    # top_k > 32
    (4, 256, 16, 128, 17, 1),    # top_k > E
    (-1, 256, 16, 128, 2, 1),    # negative batch
])
def test_workspace_size_rejects_bad_shapes(lib, B, H, E, I, k, code):
    s = binding.Shape(B, H, E, I)
    out = ctypes.c_size_t(0)
    assert lib.slimwise_moe_workspace_size(ctypes.byref(s), k, ctypes.byref(out)) == code


def _fake(addr=0x10000):
    return ctypes.c_void_p(addr)


def test_decode_rejects_bad_arguments_without_cuda(lib):
    s = binding.Shape(4, 256, 16, 128)
    big = 1 << 30
    P = _fake
    # top_k larger than the retained pool
    assert lib.slimwise_moe_decode(P(), P(), P(), 2, P(), P(), 4, P(), None, ctypes.byref(s), P(), big) == 1
    # retained pool larger than E
    assert lib.slimwise_moe_decode(P(), P(), P(), 17, P(), P(), 2, P(), None, ctypes.byref(s), P(), big) == 1
    # null retained_idx for the pruned entry point
    assert lib.slimwise_moe_decode(P(), P(), None, 8, P(), P(), 2, P(), None, ctypes.byref(s), P(), big) == 1
    # null weight
    assert lib.slimwise_moe_decode(P(), P(), P(), 8, None, P(), 2, P(), None, ctypes.byref(s), P(), big) == 1
    # misaligned hidden
    assert lib.slimwise_moe_decode(P(0x10004), P(), P(), 8, P(), P(), 2, P(), None, ctypes.byref(s), P(), big) == 2
    # workspace too small
    assert lib.slimwise_moe_decode(P(), P(), P(), 8, P(), P(), 2, P(), None, ctypes.byref(s), P(), 1024) == 3
    # misaligned workspace
    assert lib.slimwise_moe_decode(P(), P(), P(), 8, P(), P(), 2, P(), None, ctypes.byref(s), P(0x10010), big) == 2
    # null shape
    assert lib.slimwise_moe_decode(P(), P(), P(), 8, P(), P(), 2, P(), None, None, P(), big) == 1
    # B == 0 is a successful no-op, even with null buffers
    s0 = binding.Shape(0, 256, 16, 128)
    assert lib.slimwise_moe_decode(None, None, P(), 8, None, None, 2, None, None, ctypes.byref(s0), None, 0) == 0
    assert lib.slimwise_moe_decode_full(None, None, None, None, 2, None, None, ctypes.byref(s0), None, 0) == 0


def test_route_and_group_reject_bad_arguments_without_cuda(lib):
    s = binding.Shape(4, 256, 16, 128)
    P = _fake
    null8 = [None] * 8
    assert lib.slimwise_moe_route(P(), P(), P(), 8, 9, None, ctypes.byref(s), P(), 1 << 30, *null8) == 1
    assert lib.slimwise_moe_route(None, P(), P(), 8, 2, None, ctypes.byref(s), P(), 1 << 30, *null8) == 1
    assert lib.slimwise_moe_group(None, 2, None, ctypes.byref(s), P(), 1 << 30, *null8[:6]) == 1
    assert lib.slimwise_moe_group(P(), 2, None, ctypes.byref(s), P(), 16, *null8[:6]) == 3
    flags = ctypes.c_int32(0)
    assert lib.slimwise_moe_device_status(None, None, ctypes.byref(flags)) == 1


def test_binding_refuses_cpu_tensors(lib):
    import torch
    x = torch.zeros(4, 256, dtype=torch.bfloat16)
    with pytest.raises(TypeError):
        binding.slimwise_moe_decode_full(x, torch.zeros(16, 256), torch.zeros(16, 256, 256, dtype=torch.bfloat16),
                                         torch.zeros(16, 256, 128, dtype=torch.bfloat16), 2)


def test_shared_expert_entry_points_validate_without_cuda(lib):
    P = _fake
    out = ctypes.c_size_t(0)
    s64 = binding.Shape(64, 2048, 128, 768)
    # the workspace grows by the shared expert's gate, token-order hidden
    # rows, activations and outputs
    n0 = _ws(64, 2048, 128, 768, 8)
    assert lib.slimwise_moe_shared_workspace_size(ctypes.byref(s64), 8, 1024, ctypes.byref(out)) == 0
    assert out.value >= n0 + 64 * (4 + 2 * 2048 + 2 * 1024 + 2 * 2048)
    s = binding.Shape(4, 256, 16, 128)
    for bad_is in (0, 32, 96, 1 << 17):
        assert lib.slimwise_moe_shared_workspace_size(ctypes.byref(s), 2, bad_is, ctypes.byref(out)) == 2
    big = 1 << 30

    def call(gate=P(), gu=P(), dn=P(), Is=128, ws_bytes=big, shape=s):
        return lib.slimwise_moe_decode_shared(P(), P(), P(), 8, P(), P(), 2, gate, gu, dn, Is, P(),
                                              None, ctypes.byref(shape), P(), ws_bytes)

    assert call(Is=96) == 2                 # Is not a multiple of 64
    assert call(gate=None) == 1             # missing shared gate row
    assert call(dn=None) == 1               # missing shared down weight
    assert call(gate=P(0x10004)) == 2       # misaligned gate row
    assert call(ws_bytes=1024) == 3         # workspace too small
    # the plain layer's workspace is too small once a shared expert is added
    n_plain = _ws(4, 256, 16, 128, 2)
    assert call(ws_bytes=n_plain) == 3
    # B = 0 is a no-op even with null buffers
    s0 = binding.Shape(0, 256, 16, 128)
    assert lib.slimwise_moe_decode_shared(None, None, None, 0, None, None, 2, None, None, None, 128,
                                          None, None, ctypes.byref(s0), None, 0) == 0


def test_statistics_entry_points_validate_without_cuda(lib):
    P = _fake
    s = binding.Shape(4, 256, 16, 128)
    big = 1 << 30
    # null statistics buffer; misaligned one
    assert lib.slimwise_moe_expert_stats(P(), P(), P(), P(), 2, None, P(), None, ctypes.byref(s), P(), big) == 1
    assert lib.slimwise_moe_expert_stats(P(), P(), P(), P(), 2, P(0x10004), P(), None, ctypes.byref(s), P(), big) == 2
    # bad shape is reported before anything else
    bad = binding.Shape(4, 100, 16, 128)
    assert lib.slimwise_moe_expert_stats(P(), P(), P(), P(), 2, P(), P(), None, ctypes.byref(bad), P(), big) == 2
    s0 = binding.Shape(0, 256, 16, 128)
    assert lib.slimwise_moe_expert_stats(None, None, None, None, 2, None, None, None, ctypes.byref(s0), None, 0) == 0
    # selection: pool too large, m' out of range, unknown criterion, null outputs
    assert lib.slimwise_moe_select_retained(P(), 2000, 8, 2, P(), None) == 2
    assert lib.slimwise_moe_select_retained(P(), 16, 17, 2, P(), None) == 1
    assert lib.slimwise_moe_select_retained(P(), 16, 8, 3, P(), None) == 1
    assert lib.slimwise_moe_select_retained(None, 16, 8, 2, P(), None) == 1
    assert lib.slimwise_moe_select_retained(P(), 16, 0, 2, None, None) == 0


def test_compact_layer_validates_without_cuda(lib):
    P = _fake
    s = binding.Shape(0, 256, 16, 128)
    args = lambda **kw: [kw.get(n, P()) for n in ("gu", "dn", "wr", "ret")]
    out = [P(), P(), P(), P()]
    # null input or output pointers
    assert lib.slimwise_moe_compact_layer(None, P(), P(), P(), 8, ctypes.byref(s), *out, None) == 1
    assert lib.slimwise_moe_compact_layer(*args(), 8, ctypes.byref(s), P(), P(), P(), None, None) == 1
    # retained count out of [1, E]; no shape
    assert lib.slimwise_moe_compact_layer(*args(), 0, ctypes.byref(s), *out, None) == 1
    assert lib.slimwise_moe_compact_layer(*args(), 17, ctypes.byref(s), *out, None) == 1
    assert lib.slimwise_moe_compact_layer(*args(), 8, None, *out, None) == 1
    # unsupported shape; misaligned weights or ids
    bad = binding.Shape(0, 100, 16, 128)
    assert lib.slimwise_moe_compact_layer(*args(), 8, ctypes.byref(bad), *out, None) == 2
    assert lib.slimwise_moe_compact_layer(*args(gu=P(0x10008)), 8, ctypes.byref(s), *out, None) == 2
    assert lib.slimwise_moe_compact_layer(*args(ret=P(0x10002)), 8, ctypes.byref(s), *out, None) == 2
    # num_tokens is not used: with a negative one the shape error is still
    # the one reported (every call above and here fails before any CUDA call)
    neg = binding.Shape(-5, 100, 16, 128)
    assert lib.slimwise_moe_compact_layer(*args(), 8, ctypes.byref(neg), *out, None) == 2
