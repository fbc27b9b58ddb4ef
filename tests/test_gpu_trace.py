"""The timeline trace (tracing subsystem): the trace build's kernels stamp
each phase of every layer call into the workspace, and the phases must come
out in the order the pipeline runs them; the product build writes no stamps.

The library is chosen once per process, so the trace build runs in a child
process (SLIMWISE_LIBRARY), while this process keeps the product build.
"""
import json
import os
import subprocess
import sys

import pytest
import torch

import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import synth, trace

pytestmark = pytest.mark.gpu
ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

_CHILD = r"""
import json, torch
import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import synth, trace, binding
assert binding.library_path().endswith("libslimwise_trace.so")
dev = torch.device("cuda", 0)
shape = synth.QWEN
w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
wr = synth.router_weight(shape, 0, device=dev)
ret = synth.retained_set(shape.num_experts, 64, 2).to(dev)
x = synth.hidden_states(64, shape, 1, device=dev)
ws = sw.alloc_workspace(64, shape.hidden, shape.num_experts, shape.inter, shape.top_k, dev)
ws.zero_()
out = None
for i in range(6):
    out = sw.slimwise_moe_decode(x, wr, ret, w_gu, w_d, shape.top_k, out=out, workspace=ws)
torch.cuda.synchronize()
ring, nxt = trace.read_ring(ws)
print(json.dumps({"next": nxt, "timeline": trace.timeline(ws, 6)}))
"""


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()


def test_trace_build_stamps_phases_in_pipeline_order():
    path = sw.build.build(trace=True)
    env = dict(os.environ, SLIMWISE_LIBRARY=path, PYTHONPATH=ROOT)
    r = subprocess.run([sys.executable, "-c", _CHILD], env=env, cwd=ROOT, capture_output=True,
                       text=True, timeout=900)
    assert r.returncode == 0, r.stderr[-2000:]
    res = json.loads(r.stdout.strip().splitlines()[-1])
    assert res["next"] == 6                        # the step counter started from the zeroed word
    for step in res["timeline"]:
        v = [step[p] for p in trace.PHASES]
        assert v[0] == 0.0
        # each phase starts after the previous grid has finished (dependency waits)
        assert all(a <= b for a, b in zip(v, v[1:])), step
        assert 0.0 < step["ffn_end"] < 5000.0, step


def test_product_build_writes_no_stamps():
    shape = synth.TINY
    dev = torch.device("cuda", 0)
    w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
    wr = synth.router_weight(shape, 0, device=dev)
    x = synth.hidden_states(4, shape, 1, device=dev)
    ws = sw.alloc_workspace(4, shape.hidden, shape.num_experts, shape.inter, shape.top_k, dev)
    ws.zero_()
    sw.slimwise_moe_decode_full(x, wr, w_gu, w_d, shape.top_k, workspace=ws)
    ring, _ = trace.read_ring(ws)
    assert not ring.any()
