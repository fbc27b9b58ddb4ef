"""The entry point for callers that cannot allocate device memory.

slimwise_moe_decode_noalloc runs the decode layer with its scratch in a fixed
device array inside the library, for hosts (engines with all memory reserved
up front, plugins handed only inputs and outputs) that must not call
cudaMalloc.  Two calls in a row -- the second with a different batch, reusing
whatever the first left in the array -- must each match slimwise_moe_decode
(the workspace entry point) within the layer's output tolerance.  This file
is collected last so a failure here comes after every other test has run.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_34117_gb300 import binding, build, synth

pytestmark = pytest.mark.gpu

REL_L2_TOL = 1e-2
MAX_ABS_TOL = 3e-2


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def test_noalloc_entry_point_matches_workspace_entry_point_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    lib = binding.load()
    dev = torch.device("cuda")
    shape = synth.QWEN
    w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
    wr = synth.router_weight(shape, 0, device=dev)
    retained = synth.retained_set(shape.num_experts, 64, 2).to(dev)
    stream = torch.cuda.current_stream()
    for B, seed in ((64, 31), (96, 32)):
        x = synth.hidden_states(B, shape, seed, device=dev)
        ref = binding.slimwise_moe_decode(x, wr, retained, w_gu, w_d, shape.top_k)
        out = torch.full((B, shape.hidden), float("nan"), dtype=torch.bfloat16, device=dev)
        s = binding.Shape(B, shape.hidden, shape.num_experts, shape.inter)
        rc = lib.slimwise_moe_decode_noalloc(_ptr(x), _ptr(wr), _ptr(retained), int(retained.numel()),
                                             _ptr(w_gu), _ptr(w_d), shape.top_k, _ptr(out),
                                             ctypes.c_void_p(stream.cuda_stream), ctypes.byref(s))
        assert rc == 0, binding.STATUS_NAMES.get(rc, rc)
        torch.cuda.synchronize()
        got = out.double().cpu().numpy()
        want = ref.double().cpu().numpy()
        err = np.linalg.norm(got - want) / np.linalg.norm(want)
        mx = np.abs(got - want).max()
        assert err <= REL_L2_TOL and mx <= MAX_ABS_TOL, (B, err, mx)


def test_noalloc_rejects_problems_larger_than_its_scratch():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build()
    lib = binding.load()
    shape = synth.QWEN
    s = binding.Shape(1024, shape.hidden, shape.num_experts, shape.inter)
    p = ctypes.c_void_p(0x10000)
    # checked on the host before anything is launched
    assert lib.slimwise_moe_decode_noalloc(p, p, None, 0, p, p, shape.top_k, p, None, ctypes.byref(s)) == 3
