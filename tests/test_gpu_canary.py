"""Guard bytes around every buffer the library writes: a bounds check that
needs no memory-checking tool.

Each call gets its workspace and its outputs as views into larger buffers
whose leading and trailing 64 KB hold a known pattern.  A write past either
end of a buffer lands in its own guard (inside the allocation, so nothing
faults) and changes the pattern; after every call all guards must be intact.
The cases cover each shape class the kernels distinguish: routing clusters of
1 to 16 tokens, 128-row, wide and CTA-pair FFN items, split hot experts, the
shared expert, a wide hidden size and the compact checkpoint.
"""
import ctypes

import pytest
import torch

import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import binding, synth

pytestmark = pytest.mark.gpu
DEV = "cuda"
PAD = 64 * 1024          # guard bytes on each side (a multiple of 256: keeps alignment)
PATTERN = 0xA5


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()


class Guarded:
    """A uint8 buffer of `nbytes` between two guards of PAD bytes."""

    def __init__(self, nbytes):
        self.nbytes = nbytes
        self.buf = torch.full((PAD + nbytes + PAD,), PATTERN, dtype=torch.uint8, device=DEV)

    def view(self, dtype=torch.uint8, shape=None):
        v = self.buf[PAD:PAD + self.nbytes].view(dtype)
        return v if shape is None else v.view(shape)

    def intact(self):
        return bool((self.buf[:PAD] == PATTERN).all()) and bool((self.buf[PAD + self.nbytes:] == PATTERN).all())


def _layer(shape, seed):
    w_gu, w_d = synth.expert_weights(shape, seed, device=DEV)
    return w_gu, w_d, synth.router_weight(shape, seed, device=DEV)


CASES = [
    # (name, shape, B, m', extra)
    ("tiny_B1", synth.TINY, 1, 8, {}),
    ("tiny_B37", synth.TINY, 37, 8, {}),
    ("tiny_B600", synth.TINY, 600, 4, {}),
    ("generic_H640", synth.LayerShape(hidden=640, num_experts=24, inter=192, top_k=3), 33, 12, {}),
    ("wide_H8192", synth.LayerShape(hidden=8192, num_experts=16, inter=128, top_k=2), 200, 8, {}),
    ("qwen_B64_full", synth.QWEN, 64, None, {}),
    ("qwen_B256_m64_wide", synth.QWEN, 256, 64, {}),
    ("qwen_B512_m32", synth.QWEN, 512, 32, {}),
    ("qwen_B305_m32", synth.QWEN, 305, 32, {}),
    ("qwen_B256_m64_pairs", synth.QWEN, 256, 64, {"ffn_items": 1}),
    ("hot_expert", synth.LayerShape(hidden=256, num_experts=64, inter=128, top_k=2), 256, 8, {"hot": True}),
]


@pytest.mark.parametrize("name,shape,B,m_prime,extra", CASES, ids=[c[0] for c in CASES])
def test_decode_writes_stay_inside_workspace_and_output(name, shape, B, m_prime, extra):
    w_gu, w_d, wr = _layer(shape, 3)
    x = synth.hidden_states(B, shape, 4, device=DEV)
    retained = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, 5).to(DEV)
    if extra.get("hot"):
        bias = torch.zeros(shape.num_experts)
        bias[int(retained[1])] = 8.0
        x, wr = synth.apply_popularity_bias(x.cpu(), wr.cpu(), bias)
        x, wr = x.to(DEV), wr.to(DEV)
    n_ws = sw.slimwise_moe_workspace_size(B, shape.hidden, shape.num_experts, shape.inter, shape.top_k)
    ws = Guarded(n_ws)
    out = Guarded(B * shape.hidden * 2)
    for _ in range(2):   # the second call runs over the first call's workspace contents
        sw.slimwise_moe_decode_ex(x, wr, retained, w_gu, w_d, shape.top_k,
                                  out=out.view(torch.bfloat16, (B, shape.hidden)),
                                  workspace=ws.view(), ffn_items=extra.get("ffn_items", 0))
    torch.cuda.synchronize()
    assert sw.slimwise_moe_device_status(ws.view()) == 0
    assert ws.intact(), "a write left the workspace"
    assert out.intact(), "a write left the output"


def test_shared_expert_writes_stay_inside_workspace_and_output():
    shape = synth.LayerShape(hidden=256, num_experts=16, inter=128, top_k=2)
    B, Is = 130, 192
    w_gu, w_d, wr = _layer(shape, 6)
    se = [t.to(DEV) for t in synth.shared_expert(shape.hidden, Is, 7)]
    x = synth.hidden_states(B, shape, 8, device=DEV)
    retained = synth.retained_set(shape.num_experts, 8, 9).to(DEV)
    n_ws = sw.slimwise_moe_shared_workspace_size(B, shape.hidden, shape.num_experts, shape.inter,
                                                 shape.top_k, Is)
    ws = Guarded(n_ws)
    out = Guarded(B * shape.hidden * 2)
    sw.slimwise_moe_decode_shared(x, wr, retained, w_gu, w_d, shape.top_k, *se,
                                  out=out.view(torch.bfloat16, (B, shape.hidden)),
                                  workspace=ws.view())
    torch.cuda.synchronize()
    assert ws.intact() and out.intact()


def test_compact_layer_writes_stay_inside_its_outputs():
    shape = synth.QWEN
    w_gu, w_d, wr = _layer(shape, 10)
    m = 33
    retained = synth.retained_set(shape.num_experts, m, 11, shuffle=True).to(DEV)
    gu_c = Guarded(m * 2 * shape.inter * shape.hidden * 2)
    d_c = Guarded(m * shape.hidden * shape.inter * 2)
    wr_c = Guarded(m * shape.hidden * 4)
    ids_c = Guarded(m * 4)
    s = binding.Shape(0, shape.hidden, shape.num_experts, shape.inter)
    P = lambda t: ctypes.c_void_p(t.data_ptr())
    rc = sw.load().slimwise_moe_compact_layer(
        P(w_gu), P(w_d), P(wr), P(retained), m, ctypes.byref(s), P(gu_c.view()), P(d_c.view()),
        P(wr_c.view()), P(ids_c.view()), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0
    torch.cuda.synchronize()
    assert all(g.intact() for g in (gu_c, d_c, wr_c, ids_c))
    ids = torch.sort(retained.long()).values
    assert torch.equal(gu_c.view(torch.bfloat16, (m, 2 * shape.inter, shape.hidden)),
                       w_gu.index_select(0, ids))
