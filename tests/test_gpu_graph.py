"""The layer captured in a CUDA graph and replayed gives the eager calls'
outputs bit for bit.

A serving engine records a decode step once and replays it; the layer's
launches (four kernels chained with programmatic dependent launch, their TMA
descriptors passed by value) must replay correctly with new inputs copied
into the captured buffers.  The kernels are deterministic, so the replayed
outputs must equal the eager ones exactly.
"""
import pytest
import torch

import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import synth

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()


def _layer(shape, seed, m_prime):
    w_gu, w_d = synth.expert_weights(shape, seed, device=DEV)
    wr = synth.router_weight(shape, seed, device=DEV)
    ret = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, seed + 1).to(DEV)
    return w_gu, w_d, wr, ret


def test_two_layer_step_replays_bit_exactly():
    big, small = synth.QWEN, synth.TINY
    B = 64
    L1 = _layer(big, 0, 64)            # pruned Qwen-class layer
    L2 = _layer(small, 3, None)        # a second, different layer: full tiny pool
    k1, k2 = big.top_k, small.top_k
    ws1 = sw.alloc_workspace(B, big.hidden, big.num_experts, big.inter, k1, DEV)
    ws2 = sw.alloc_workspace(B, small.hidden, small.num_experts, small.inter, k2, DEV)
    batches = [(synth.hidden_states(B, big, 10 + i, device=DEV),
                synth.hidden_states(B, small, 20 + i, device=DEV)) for i in range(3)]

    def step(x1, x2, o1, o2, stream):
        w_gu, w_d, wr, ret = L1
        sw.slimwise_moe_decode_ex(x1, wr, ret, w_gu, w_d, k1, out=o1, workspace=ws1, stream=stream)
        w_gu, w_d, wr, _ = L2
        sw.slimwise_moe_decode_ex(x2, wr, None, w_gu, w_d, k2, out=o2, workspace=ws2, stream=stream)

    # eager reference outputs
    eager = []
    for x1, x2 in batches:
        o1 = torch.empty((B, big.hidden), dtype=torch.bfloat16, device=DEV)
        o2 = torch.empty((B, small.hidden), dtype=torch.bfloat16, device=DEV)
        step(x1, x2, o1, o2, torch.cuda.current_stream())
        eager.append((o1, o2))
    torch.cuda.synchronize()

    # capture once on static buffers, replay with each batch copied in
    sx1, sx2 = torch.empty_like(batches[0][0]), torch.empty_like(batches[0][1])
    so1 = torch.empty((B, big.hidden), dtype=torch.bfloat16, device=DEV)
    so2 = torch.empty((B, small.hidden), dtype=torch.bfloat16, device=DEV)
    sx1.copy_(batches[0][0])
    sx2.copy_(batches[0][1])
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        step(sx1, sx2, so1, so2, side)      # warm-up outside the capture (encodes the maps)
        side.synchronize()
        with torch.cuda.graph(g, stream=side):
            step(sx1, sx2, so1, so2, side)
    torch.cuda.current_stream().wait_stream(side)
    for rep in range(2):
        for (x1, x2), (e1, e2) in zip(batches, eager):
            sx1.copy_(x1)
            sx2.copy_(x2)
            g.replay()
            torch.cuda.synchronize()
            assert torch.equal(so1, e1), rep
            assert torch.equal(so2, e2), rep
    assert sw.slimwise_moe_device_status(ws1) == 0
    assert sw.slimwise_moe_device_status(ws2) == 0
