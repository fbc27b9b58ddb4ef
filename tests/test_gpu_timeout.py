"""A bounded device wait that runs out: failure detection without a GPU fault.

Every wait of the expert-FFN kernel has a time limit.  The test-only launch
option test_starve_first_down makes the first routed down item wait for one
gate/up tile more than exists, with a short wait_limit_ns, so that wait must
run out.  The call then records SLIMWISE_DEVERR_DEPENDENCY_TIMEOUT; the CTA
that gave up drains its copies and MMAs, frees its tensor memory and exits,
and the kernel completes well before the default 1 s limit.  The next normal
call on the same workspace must read a clear error word and match the oracle
(the GPU stays usable).
"""
import time

import numpy as np
import pytest
import torch

import oracle
import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import synth

pytestmark = pytest.mark.gpu

DEV = "cuda"
WAIT_LIMIT_NS = 2_000_000   # 2 ms: far above any legitimate wait of a tiny layer


@pytest.fixture(scope="module")
def tiny():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()
    oracle.build()
    shape = synth.TINY
    w_gu, w_d = synth.expert_weights(shape, 0)
    wr = synth.router_weight(shape, 0)
    return shape, w_gu, w_d, wr


# (8, 2): one work entry per expert; (300, 8): two entries per expert, so
# the starved item's entry shares its expert with a running one
@pytest.mark.parametrize("B,k", [(8, 2), (300, 8)])
def test_dependency_wait_runs_out_and_next_call_is_clean(tiny, B, k):
    shape, w_gu, w_d, wr = tiny
    x = synth.hidden_states(B, shape, 90 + B)
    ret = synth.retained_set(shape.num_experts, 8, 2)
    xd, wrd, retd = x.to(DEV), wr.to(DEV), ret.to(DEV)
    gud, dnd = w_gu.to(DEV), w_d.to(DEV)
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    sw.slimwise_moe_decode_ex(xd, wrd, retd, gud, dnd, k, workspace=ws, wait_limit_ns=WAIT_LIMIT_NS,
                              test_starve_first_down=True)
    flags = sw.slimwise_moe_device_status(ws)       # synchronises the stream
    elapsed = time.perf_counter() - t0
    assert flags & sw.binding.DEVERR_DEPENDENCY_TIMEOUT, flags
    assert not flags & (sw.binding.DEVERR_DUPLICATE_RETAINED | sw.binding.DEVERR_BAD_RETAINED)
    assert elapsed < 0.5, elapsed                   # the short limit, not the default 1 s
    # the same workspace, a normal call: clear error word, oracle results
    out = sw.slimwise_moe_decode(xd, wrd, retd, gud, dnd, k, workspace=ws)
    assert sw.slimwise_moe_device_status(ws) == 0
    route = sw.slimwise_moe_route(xd, wrd, retd, k, shape.num_experts, shape.inter)
    torch.cuda.synchronize()
    ref = oracle.moe_decode(synth.bf16_bits(x), wr.numpy(), ret.numpy(), synth.bf16_bits(w_gu),
                            synth.bf16_bits(w_d), k)
    assert np.array_equal(route["topk_idx"].cpu().numpy(), ref["idx"])
    got = out.double().cpu().numpy()
    err = np.linalg.norm(got - ref["out"]) / np.linalg.norm(ref["out"])
    assert err <= 1e-2 and np.abs(got - ref["out"]).max() <= 3e-2, err
    # and the default limit still lets a normal call with the option off finish
    out2 = sw.slimwise_moe_decode_ex(xd, wrd, retd, gud, dnd, k, workspace=ws,
                                     wait_limit_ns=WAIT_LIMIT_NS)
    assert sw.slimwise_moe_device_status(ws) == 0
    assert torch.equal(out2, out)
