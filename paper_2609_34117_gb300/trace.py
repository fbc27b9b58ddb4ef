"""Timeline of one decode layer's kernels, from the trace build of the library.

`build.build(trace=True)` compiles the same kernels with %globaltimer stamps
(SLIMWISE_TRACE).  They go into a ring of 16 steps that follows the control
words at the head of the workspace, one step per layer call:

    route_start, route_end    routing grid, first CTA: after its dependency
                              wait, and when it finishes
    group_start, group_end    grouping grid, first CTA, likewise
    ffn_start                 expert-FFN grid, first CTA after its wait
    ffn_first_data            first stage of weights and tokens in that CTA
    ffn_end                   the FFN grid's last CTA to finish

A process selects the trace build with SLIMWISE_LIBRARY=<build.TRACE_LIB_PATH>
(the library is chosen once per process, at its first call).  The stamps do
not change any result.

    python -m paper_2609_34117_gb300.trace [--batch 64] [--retained 128]

runs the Qwen-class layer with the trace build and prints the median offset
of each phase from the routing start, in microseconds.
"""
from __future__ import annotations

import numpy as np
import torch

# Layout of the workspace head (common.cuh): 16 int32 control words, the
# trace-step counter among them, then the ring of [16 steps][8 slots] uint64.
CTRL_WORDS = 16
TRACE_STEP_WORD = 6
TRACE_STEPS = 16
TRACE_SLOTS = 8
PHASES = ("route_start", "route_end", "group_start", "group_end", "ffn_start",
          "ffn_first_data", "ffn_end")


def read_ring(workspace: torch.Tensor):
    """(stamps uint64 [16, 8] in ns, next step number) from a workspace of
    the trace build; synchronises the workspace's device."""
    head = workspace[: CTRL_WORDS * 4 + TRACE_STEPS * TRACE_SLOTS * 8].cpu().numpy()
    ctrl = head[: CTRL_WORDS * 4].view(np.int32)
    ring = head[CTRL_WORDS * 4:].view(np.uint64).reshape(TRACE_STEPS, TRACE_SLOTS)
    return ring, int(ctrl[TRACE_STEP_WORD])


def timeline(workspace: torch.Tensor, steps: int):
    """The last `steps` (<= 16) layer calls made on this workspace, oldest
    first: one dict per call with each phase's offset from its routing start
    in microseconds (route_start = 0)."""
    if not 1 <= steps <= TRACE_STEPS:
        raise ValueError(f"steps must be in [1, {TRACE_STEPS}]")
    ring, nxt = read_ring(workspace)
    out = []
    for s in range(nxt - steps, nxt):
        row = ring[s % TRACE_STEPS].astype(np.int64)
        t0 = row[0]
        out.append({p: (int(row[i]) - int(t0)) / 1e3 for i, p in enumerate(PHASES)})
    return out


def _main():
    import argparse
    import os
    import sys

    from . import build, synth

    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--batch", type=int, default=64)
    ap.add_argument("--retained", type=int, default=128)
    ap.add_argument("--calls", type=int, default=16)
    args = ap.parse_args()
    path = build.build(trace=True)
    if os.environ.get("SLIMWISE_LIBRARY") != path:
        # the library is fixed at a process's first call: start one that loads the trace build
        env = dict(os.environ, SLIMWISE_LIBRARY=path)
        os.execve(sys.executable, [sys.executable, "-m", "paper_2609_34117_gb300.trace",
                                   *sys.argv[1:]], env)
    from . import binding as sw
    dev = torch.device("cuda", 0)
    shape = synth.QWEN
    w_gu, w_d = synth.expert_weights(shape, 0, device=dev)
    wr = synth.router_weight(shape, 0, device=dev)
    ret = (None if args.retained >= shape.num_experts
           else synth.retained_set(shape.num_experts, args.retained, 2).to(dev))
    xs = [synth.hidden_states(args.batch, shape, 1 + j, device=dev) for j in range(8)]
    ws = sw.alloc_workspace(args.batch, shape.hidden, shape.num_experts, shape.inter,
                            shape.top_k, dev)
    out = torch.empty((args.batch, shape.hidden), dtype=torch.bfloat16, device=dev)
    for i in range(64 + args.calls):
        sw.slimwise_moe_decode_ex(xs[i % 8], wr, ret, w_gu, w_d, shape.top_k, out=out,
                                  workspace=ws)
    torch.cuda.synchronize()
    tl = timeline(ws, min(args.calls, TRACE_STEPS))
    med = {p: float(np.median([t[p] for t in tl])) for p in PHASES}
    print(" ".join(f"{p}={med[p]:.1f}" for p in PHASES))


if __name__ == "__main__":
    _main()
