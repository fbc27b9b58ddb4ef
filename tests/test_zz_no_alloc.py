"""The entry point for callers that cannot allocate device memory.

slimwise_moe_decode_noalloc runs the decode layer with its scratch in a fixed
device array inside the library, for hosts (engines with all memory reserved
up front, plugins handed only inputs and outputs) that must not call
cudaMalloc.  Consecutive calls reuse whatever the previous call left in the
array: the batch grows, then shrinks to a few tokens on the full pool, and
every call must give exactly the output of slimwise_moe_decode (the workspace
entry point runs the same deterministic kernels).  One call is also checked
against the CPU oracle, and the array's error word is read back through
slimwise_moe_noalloc_device_status.  This file is collected last so a failure
here comes after every other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2609_34117_gb300 import binding, build, synth

pytestmark = pytest.mark.gpu

REL_L2_TOL = 1e-2
MAX_ABS_TOL = 3e-2


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _noalloc(lib, x, wr, retained, w_gu, w_d, shape):
    B = x.shape[0]
    out = torch.full((B, shape.hidden), float("nan"), dtype=torch.bfloat16, device=x.device)
    s = binding.Shape(B, shape.hidden, shape.num_experts, shape.inter)
    n_ret = 0 if retained is None else int(retained.numel())
    stream = torch.cuda.current_stream()
    rc = lib.slimwise_moe_decode_noalloc(_ptr(x), _ptr(wr), _ptr(retained), n_ret, _ptr(w_gu),
                                         _ptr(w_d), shape.top_k, _ptr(out),
                                         ctypes.c_void_p(stream.cuda_stream), ctypes.byref(s))
    assert rc == 0, binding.STATUS_NAMES.get(rc, rc)
    return out


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    oracle.build()
    return binding.load()


def test_noalloc_entry_point_matches_workspace_entry_point_on_reuse(lib):
    dev = torch.device("cuda")
    shape = synth.QWEN
    w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
    wr = synth.router_weight(shape, 0, device=dev)
    pool64 = synth.retained_set(shape.num_experts, 64, 2).to(dev)
    # grow the batch, then shrink it to 8 tokens over the full pool: stale
    # counts, entries or union ids of a larger earlier call must not leak
    calls = ((64, 31, pool64), (96, 32, pool64), (8, 33, None))
    outs = []
    for B, seed, retained in calls:
        x = synth.hidden_states(B, shape, seed, device=dev)
        out = _noalloc(lib, x, wr, retained, w_gu, w_d, shape)
        if retained is None:
            ref = binding.slimwise_moe_decode_full(x, wr, w_gu, w_d, shape.top_k)
        else:
            ref = binding.slimwise_moe_decode(x, wr, retained, w_gu, w_d, shape.top_k)
        torch.cuda.synchronize()
        assert binding.slimwise_moe_noalloc_device_status() == 0
        assert torch.equal(out, ref), B
        outs.append((x, retained, out))
    # the 8-token full-pool call against the oracle, every token
    x, _, out = outs[2]
    want = oracle.moe_decode(synth.bf16_bits(x), wr.cpu().numpy(), None, synth.bf16_bits(w_gu),
                             synth.bf16_bits(w_d), shape.top_k)["out"]
    got = out.double().cpu().numpy()
    err = np.linalg.norm(got - want) / np.linalg.norm(want)
    assert err <= REL_L2_TOL and np.abs(got - want).max() <= MAX_ABS_TOL, err


def test_noalloc_status_reports_device_errors(lib):
    dev = torch.device("cuda")
    shape = synth.TINY
    w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
    wr = synth.router_weight(shape, 0, device=dev)
    x = synth.hidden_states(4, shape, 4, device=dev)
    # a repeated retained id is reported in the array's error word
    dup = torch.tensor([1, 3, 3, 7, 9], dtype=torch.int32, device=dev)
    _noalloc(lib, x, wr, dup, w_gu, w_d, shape)
    flags = binding.slimwise_moe_noalloc_device_status()
    assert flags & binding.DEVERR_DUPLICATE_RETAINED, flags
    # the next clean call starts from a cleared word
    ok = torch.tensor([1, 3, 7, 9], dtype=torch.int32, device=dev)
    out = _noalloc(lib, x, wr, ok, w_gu, w_d, shape)
    assert binding.slimwise_moe_noalloc_device_status() == 0
    ref = binding.slimwise_moe_decode(x, wr, ok, w_gu, w_d, shape.top_k)
    torch.cuda.synchronize()
    assert torch.equal(out, ref)


def test_noalloc_rejects_problems_larger_than_its_scratch(lib):
    shape = synth.QWEN
    s = binding.Shape(1024, shape.hidden, shape.num_experts, shape.inter)
    p = ctypes.c_void_p(0x10000)
    # checked on the host before anything is launched
    assert lib.slimwise_moe_decode_noalloc(p, p, None, 0, p, p, shape.top_k, p, None, ctypes.byref(s)) == 3
