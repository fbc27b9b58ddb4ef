"""The tracing subsystem without a GPU: the trace build compiles and exports
the same C ABI, the Python reader's layout constants are the ones the
kernels use, and the reader turns a ring of stamps into per-call offsets
(including a ring that has wrapped)."""
import os
import re

import numpy as np
import torch

from paper_2609_34117_gb300 import binding, build, trace

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _common_cuh():
    with open(os.path.join(ROOT, "paper_2609_34117_gb300", "csrc", "common.cuh")) as f:
        return f.read()


def test_reader_layout_matches_the_kernels():
    src = _common_cuh()
    assert int(re.search(r"kCtrlWords\s*=\s*(\d+)", src).group(1)) == trace.CTRL_WORDS
    assert int(re.search(r"kCtrlTraceStep\s*=\s*(\d+)", src).group(1)) == trace.TRACE_STEP_WORD
    assert int(re.search(r"kTraceSteps\s*=\s*(\d+)", src).group(1)) == trace.TRACE_STEPS
    assert int(re.search(r"kTrSlots\s*=\s*(\d+)", src).group(1)) == trace.TRACE_SLOTS
    # the slot order of the TraceSlot enum is the reader's phase order
    body = re.search(r"enum TraceSlot\s*\{(.*?)\};", src, re.S).group(1)
    names = [n.split("=")[0].strip() for n in body.replace("\n", " ").split(",")]
    names = [n for n in names if n and n != "kTrSlots"]
    expect = ["kTrRouteStart", "kTrRouteEnd", "kTrGroupStart", "kTrGroupEnd", "kTrFfnStart",
              "kTrFfnFirstData", "kTrFfnEnd"]
    assert names == expect
    assert len(trace.PHASES) == len(expect)


def _workspace_with(stamps_by_step, next_step):
    ws = torch.zeros(trace.CTRL_WORDS * 4 + trace.TRACE_STEPS * trace.TRACE_SLOTS * 8 + 64,
                     dtype=torch.uint8)
    ctrl = ws[: trace.CTRL_WORDS * 4].view(torch.int32)
    ctrl[trace.TRACE_STEP_WORD] = next_step
    ring = ws[trace.CTRL_WORDS * 4: trace.CTRL_WORDS * 4 + trace.TRACE_STEPS * trace.TRACE_SLOTS * 8]
    ring = ring.view(torch.int64).view(trace.TRACE_STEPS, trace.TRACE_SLOTS)
    for step, row in stamps_by_step.items():
        ring[step % trace.TRACE_STEPS, : len(row)] = torch.tensor(row, dtype=torch.int64)
    return ws


def test_timeline_offsets_across_a_wrapped_ring():
    base = 10_000_000_000
    stamps = {}
    for step in range(14, 20):             # steps 14..19 occupy ring slots 14, 15, 0, 1, 2, 3
        t0 = base + step * 200_000
        stamps[step] = [t0, t0 + 4_000, t0 + 5_000, t0 + 10_000, t0 + 11_000, t0 + 13_000,
                        t0 + 58_000 + step]
    ws = _workspace_with(stamps, next_step=20)
    tl = trace.timeline(ws, 6)
    assert len(tl) == 6
    for i, step in enumerate(range(14, 20)):
        assert tl[i]["route_start"] == 0.0
        assert tl[i]["route_end"] == 4.0
        assert tl[i]["ffn_first_data"] == 13.0
        assert abs(tl[i]["ffn_end"] - (58.0 + step / 1e3)) < 1e-9
    try:
        trace.timeline(ws, 17)
    except ValueError:
        pass
    else:
        raise AssertionError("more steps than the ring holds must be refused")


def test_library_override_and_trace_build_exports_the_abi(monkeypatch):
    monkeypatch.setenv("SLIMWISE_LIBRARY", "/nonexistent/libslimwise_trace.so")
    assert binding.library_path() == "/nonexistent/libslimwise_trace.so"
    monkeypatch.delenv("SLIMWISE_LIBRARY")
    assert binding.library_path() == build.LIB_PATH
    # the trace build compiles (its stamp code exists only under SLIMWISE_TRACE)
    # and exports every entry point of the header, like the product build
    import ctypes
    path = build.build(trace=True)
    assert path == build.TRACE_LIB_PATH and os.path.exists(path)
    lib = ctypes.CDLL(path)
    for name in binding.EXPORTED:
        assert hasattr(lib, name), name
