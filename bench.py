"""Benchmark of the pruned-pool batched-decode MoE layer on GB300.

One step = one decode MoE layer (route/top-k -> group/gather -> expert FFN +
combine) over one batch of synthetic hidden states, through the C ABI.

Default workload: the Qwen-class layer with the full pool, H=2048, E=128,
I=768, top-8, decode batch 64 (1.19 GB of touched expert weights per step,
larger than the 129 MB L2).  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl slimwise|reference]
                  [--workload qwen_full_b64|qwen_p50_b64|... (see WORKLOADS)]
                  [--sweep] [--stack40]

Under torchrun (N > 1) every rank runs an independent replica of the layer on
its own GPU (the layer has no cross-GPU exchange); value = tokens of all ranks
divided by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2609_34117_gb300 import synth  # noqa: E402

METRIC = "MoE decode-layer tokens/s; touched-expert HBM GB/s as fraction of ~8 TB/s peak"
NOMINAL_HBM_GBS = 8000.0
L2_BYTES = 129 * 1024 * 1024
SHAPES = {"qwen": synth.QWEN, "qwen36": synth.QWEN36}
WORKLOADS = {
    "qwen_full_b64": dict(B=64, m_prime=128),
    "qwen_p50_b64": dict(B=64, m_prime=64),
    "qwen_p50_b128": dict(B=128, m_prime=64),
    "qwen_p50_b256": dict(B=256, m_prime=64),
    "qwen_p75_b64": dict(B=64, m_prime=32),
    # the sweep's largest batch at 75 % pruning: 128 tokens per expert, where
    # the grid-wide combine queue and 16-token routing clusters are in use
    "qwen_p75_b512": dict(B=512, m_prime=32),
    # the same 50 % pool as a compact checkpoint holding only the retained
    # experts (full-pool entry point on [m', ...] tensors)
    "qwen_compact_p50_b64": dict(B=64, m_prime=64, compact=True),
    # Qwen3.6-shaped layer (E 256, I 512) at 25 / 50 / 75 % pruning
    "qwen36_p25_b64": dict(B=64, m_prime=192, shape="qwen36"),
    "qwen36_p50_b64": dict(B=64, m_prime=128, shape="qwen36"),
    "qwen36_p75_b64": dict(B=64, m_prime=64, shape="qwen36"),
    # the same with the distilled decoder's shared expert (Sec. 3.3): one
    # always-on expert of twice the original width (2 x 512) under a sigmoid gate
    "qwen36_se_p50_b64": dict(B=64, m_prime=128, shape="qwen36", shared=1024),
    "qwen36_se_p75_b64": dict(B=64, m_prime=64, shape="qwen36", shared=1024),
}
N_BATCHES = 8  # distinct hidden batches rotated through the timed steps


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ---------------------------------------------------------------- distributed
def dist_init():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if ws > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return ws, rank, local


def dist_barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def dist_max(ws, v: float) -> float:
    if ws <= 1:
        return v
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate(ws, per_rank_tokens: int, per_rank_seconds: float):
    """(total tokens over ranks, max seconds over ranks)."""
    return per_rank_tokens * ws, dist_max(ws, per_rank_seconds)


# ---------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.idx = device_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "100"]
        bus = _pci_bus_id(self.idx)
        if bus:
            cmd += ["-i", bus]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.reader = threading.Thread(target=self._read, daemon=True)
            self.reader.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.reader.join(timeout=2)
        return False

    def summary(self, max_mhz_hint=None):
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": max_mhz_hint, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def _pci_bus_id(idx):
    try:
        p = torch.cuda.get_device_properties(idx)
        dom, bus, devid = p.pci_domain_id, p.pci_bus_id, p.pci_device_id
        return f"{dom:08X}:{bus:02X}:{devid:02X}.0"
    except Exception:
        return None


# ---------------------------------------------------------------- inputs
class LayerInputs:
    def __init__(self, shape, seed, device, copies=1, shared=0):
        self.shape = shape
        self.copies = []
        for c in range(copies):
            w_gu, w_d = synth.expert_weights(shape, seed + 7919 * c, device=device)
            self.copies.append((w_gu, w_d))
        self.wr = synth.router_weight(shape, seed, device=device)
        # shared expert (gate row, gate/up, down) or None
        self.shared = synth.shared_expert(shape.hidden, shared, seed + 101, device=device) if shared else None

    def shared_bytes(self):
        """bf16 weight bytes of the shared expert (read every step)."""
        if self.shared is None:
            return 0
        return 2 * (self.shared[1].numel() + self.shared[2].numel())

    def workspace(self, sw, B, device):
        s = self.shape
        if self.shared is None:
            return sw.alloc_workspace(B, s.hidden, s.num_experts, s.inter, s.top_k, device)
        n = sw.slimwise_moe_shared_workspace_size(B, s.hidden, s.num_experts, s.inter, s.top_k,
                                                  self.shared[1].shape[0] // 2)
        return torch.empty(n, dtype=torch.uint8, device=device)

    def call(self, sw, x, retained, w_gu, w_d, out, ws_buf, stream, ffn_events=None):
        """One layer call through the C ABI."""
        k = self.shape.top_k
        if self.shared is None:
            sw.slimwise_moe_decode_ex(x, self.wr, retained, w_gu, w_d, k, out=out, workspace=ws_buf,
                                      stream=stream, ffn_events=ffn_events, ffn_items=FFN_ITEMS)
        else:
            sw.slimwise_moe_decode_shared(x, self.wr, retained, w_gu, w_d, k, *self.shared, out=out,
                                          workspace=ws_buf, stream=stream, ffn_events=ffn_events)

    def compacted(self, m_prime, seed_imp=2):
        """The layer as a compact checkpoint of its m' retained experts."""
        from paper_2609_34117_gb300 import checkpoint
        ret = synth.retained_set(self.shape.num_experts, m_prime, seed_imp).to(self.wr.device)
        c = LayerInputs.__new__(LayerInputs)
        c.shape = synth.LayerShape(self.shape.hidden, m_prime, self.shape.inter, self.shape.top_k)
        c.shared = self.shared
        c.copies = []
        for (w_gu, w_d) in self.copies:
            gu_c, d_c, wr_c, _ = checkpoint.compact_layer(w_gu, w_d, self.wr, ret)
            c.copies.append((gu_c, d_c))
        c.wr = wr_c
        return c

    def expert_bytes(self):
        return self.shape.expert_bytes


def kernel_source_hash():
    """Hash of the FFN kernel's sources with comments and whitespace removed, so
    that profiled counters stay attached to the code they were taken on."""
    h = hashlib.sha256()
    for name in ("expert_ffn.cu", "common.cuh"):
        with open(os.path.join(ROOT, "paper_2609_34117_gb300", "csrc", name)) as f:
            src = f.read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        src = re.sub(r"//[^\n]*", "", src)
        h.update("".join(src.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """Per-launch DRAM bytes of the expert-FFN kernel from the committed ncu summary,
    or None when the kernel changed since the capture."""
    p = os.path.join(ROOT, "profiles", "expert_ffn_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    if d.get("kernel_source_hash") != kernel_source_hash():
        return None
    return d.get("per_launch_bytes", {}).get(workload)


# ---------------------------------------------------------------- GPU arm
def run_layer_steps(sw, layer, hidden_batches, retained, k, steps, stream, ws_buf, out, copy_for_step,
                    ffn_events=None):
    for i in range(steps):
        w_gu, w_d = layer.copies[copy_for_step(i)]
        x = hidden_batches[i % len(hidden_batches)]
        ev = None if ffn_events is None else ffn_events[i]
        layer.call(sw, x, retained, w_gu, w_d, out, ws_buf, stream, ffn_events=ev)


def union_sizes(sw, layer, hidden_batches, retained, k):
    us = []
    for x in hidden_batches:
        r = sw.slimwise_moe_route(x, layer.wr, retained, k, layer.shape.num_experts, layer.shape.inter)
        us.append(int(r["union_size"].item()))
    return us


def measure_point(sw, layer, B, m_prime, steps, warmup, device, seed_x, sampler=None, soak_s=0.0):
    """Time `steps` layer calls; returns a dict of derived numbers.

    soak_s: seconds of the same layer calls run between the warm-up and the
    timed steps (untimed), so that the clock sampler around the call sees the
    GPU under this load for many samples even when K is small.
    """
    shape = layer.shape
    k = shape.top_k
    batches = [synth.hidden_states(B, shape, seed_x + j, device=device) for j in range(N_BATCHES)]
    retained = None if m_prime >= shape.num_experts else synth.retained_set(
        shape.num_experts, m_prime, 2).to(device)
    ws_buf = layer.workspace(sw, B, device)
    out = torch.empty((B, shape.hidden), dtype=torch.bfloat16, device=device)
    us = union_sizes(sw, layer, batches, retained, k)
    u_mean = float(np.mean(us))
    touched = u_mean * shape.expert_bytes + layer.shared_bytes()
    ncopies = len(layer.copies)
    rotate = touched < 4 * L2_BYTES and ncopies > 1
    copy_for_step = (lambda i: i % ncopies) if rotate else (lambda i: 0)
    stream = torch.cuda.current_stream()
    run_layer_steps(sw, layer, batches, retained, k, warmup, stream, ws_buf, out, copy_for_step)
    torch.cuda.synchronize()
    t_soak = time.perf_counter()
    while time.perf_counter() - t_soak < soak_s:
        run_layer_steps(sw, layer, batches, retained, k, 200, stream, ws_buf, out, copy_for_step)
        torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0.record(stream)
    run_layer_steps(sw, layer, batches, retained, k, steps, stream, ws_buf, out, copy_for_step)
    t1.record(stream)
    torch.cuda.synchronize()
    step_ms = t0.elapsed_time(t1) / steps
    # expert-FFN kernel alone, events on the launch stream (at least 400
    # launches whatever K is, so the clock sampler sees the GPU under load)
    ksteps = max(400, min(steps, 1000))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(ksteps)]
    for a, b in evs:   # torch creates the CUDA event on its first record
        a.record(stream)
        b.record(stream)
    torch.cuda.synchronize()
    run_layer_steps(sw, layer, batches, retained, k, ksteps, stream, ws_buf, out, copy_for_step, ffn_events=evs)
    torch.cuda.synchronize()
    ffn_ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
    # spread: events around blocks of 10 consecutive layer calls (an event
    # between every two calls would block the programmatic launch overlap)
    block = 10
    nblocks = max(40, min(steps // block, 100))
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(nblocks + 1)]
    for ev in marks:
        ev.record(stream)
    torch.cuda.synchronize()
    marks[0].record(stream)
    for bi in range(nblocks):
        run_layer_steps(sw, layer, batches, retained, k, block, stream, ws_buf, out, copy_for_step)
        marks[bi + 1].record(stream)
    torch.cuda.synchronize()
    per_step = np.array([marks[i].elapsed_time(marks[i + 1]) / block for i in range(nblocks)])
    flags = sw.slimwise_moe_device_status(ws_buf)
    if flags:
        raise RuntimeError(f"device error bits {flags:#x}")
    ffn_bytes = touched + 2 * B * shape.hidden * 2          # union weights + hidden in + out
    layer_bytes = touched + m_prime * shape.hidden * 4 + 2 * B * shape.hidden * 2
    if layer.shared is not None:
        layer_bytes += shape.hidden * 4  # shared-expert gate row
    return {
        "B": B, "m_prime": m_prime, "union_mean": u_mean, "union_eq1": m_prime * (1 - (1 - k / m_prime) ** B),
        "step_ms": step_ms, "tokens_per_s": B / (step_ms * 1e-3),
        "ffn_ms": ffn_ms, "ffn_algo_bytes": ffn_bytes, "layer_algo_bytes": layer_bytes,
        "touched_gbs": touched / (step_ms * 1e-3) / 1e9,
        "ffn_gbs": ffn_bytes / (ffn_ms * 1e-3) / 1e9,
        "weight_copies_rotated": ncopies if rotate else 1,
        "step_ms_p10": float(np.percentile(per_step, 10)),
        "step_ms_p50": float(np.percentile(per_step, 50)),
        "step_ms_p90": float(np.percentile(per_step, 90)),
        "_state": (batches, retained, ws_buf, out, copy_for_step),
    }


def graph_measure(sw, layer, B, point, calls=20, reps=50):
    """The same layer calls captured once in a CUDA graph (programmatic launch
    dependencies become graph edges) and replayed; ms per layer call."""
    batches, retained, ws_buf, out, copy_for_step = point["_state"]
    k = layer.shape.top_k
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    try:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(side):
            with torch.cuda.graph(g, stream=side):
                run_layer_steps(sw, layer, batches, retained, k, calls, side, ws_buf, out, copy_for_step)
        torch.cuda.current_stream().wait_stream(side)
        stream = torch.cuda.current_stream()
        for _ in range(3):
            g.replay()
        torch.cuda.synchronize()
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(reps):
            g.replay()
        t1.record(stream)
        torch.cuda.synchronize()
        ms = t0.elapsed_time(t1) / (reps * calls)
        return {"ms_per_step": ms, "tokens_per_s": B / (ms * 1e-3), "calls_per_graph": calls,
                "replays": reps}
    except Exception as exc:  # report, do not fail the bench line
        torch.cuda.synchronize()
        return {"error": f"{type(exc).__name__}: {exc}"[:200]}


def e2e_measure(sw, layer, B, m_prime, steps, device, point):
    """Same metric through the C ABI with host buffers: every step copies its
    batch from pinned host memory to the device, runs the layer and copies the
    output back, all inside the timed region.  As a serving loop would, the
    copies run on a copy stream with two device buffers each way, so the
    input of step i+1 and the output of step i move while step i computes."""
    shape = layer.shape
    batches, retained, ws_buf, out, copy_for_step = point["_state"]
    host_in = [b.cpu().pin_memory() for b in batches]
    host_out = [torch.empty((B, shape.hidden), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    dev_in = [torch.empty_like(batches[0]) for _ in range(2)]
    dev_out = [torch.empty_like(out) for _ in range(2)]
    st = torch.cuda.current_stream()
    cs = torch.cuda.Stream(device=device)
    ev = lambda: torch.cuda.Event()  # noqa: E731
    ev_in, ev_done, ev_out = [ev(), ev()], [ev(), ev()], [ev(), ev()]

    def h2d(i):
        j = i % 2
        cs.wait_event(ev_done[j])           # the layer that read dev_in[j] is done
        with torch.cuda.stream(cs):
            dev_in[j].copy_(host_in[i % len(host_in)], non_blocking=True)
        ev_in[j].record(cs)

    def layer_step(i):
        j = i % 2
        st.wait_event(ev_in[j])             # this step's batch is on the device
        st.wait_event(ev_out[j])            # dev_out[j] was copied out
        w_gu, w_d = layer.copies[copy_for_step(i)]
        layer.call(sw, dev_in[j], retained, w_gu, w_d, dev_out[j], ws_buf, st)
        ev_done[j].record(st)

    def d2h(i):
        j = i % 2
        cs.wait_event(ev_done[j])
        with torch.cuda.stream(cs):
            host_out[j].copy_(dev_out[j], non_blocking=True)
        ev_out[j].record(cs)

    def run(n):
        h2d(0)
        for i in range(n):
            if i + 1 < n:
                h2d(i + 1)
            layer_step(i)
            d2h(i)

    run(5)
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(cs)                           # before the first input copy
    run(steps)
    st.wait_stream(cs)                      # after the last output copy
    t1.record(st)
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / steps
    return {"value": B / (ms * 1e-3), "unit": "tokens/s", "ms_per_step": ms,
            "h2d_bytes_per_step": B * shape.hidden * 2, "d2h_bytes_per_step": B * shape.hidden * 2,
            "copies": "pinned host buffers, copy stream overlapped with compute (double-buffered)"}


def cpu_baseline(layer, B, m_prime, budget_s=15.0):
    """The CPU oracle as it stands, single-threaded, on a bounded sample of the
    workload: routing of the whole batch plus the expert FFNs of as many tokens
    as fit in about `budget_s` seconds.  Returns tokens/s."""
    import oracle
    oracle.build()
    shape = layer.shape
    w_gu, w_d = layer.copies[0]
    gu = synth.bf16_bits(w_gu)
    dn = synth.bf16_bits(w_d)
    wr = layer.wr.cpu().numpy()
    x = synth.bf16_bits(synth.hidden_states(B, shape, 1))
    ret = None if m_prime >= shape.num_experts else synth.retained_set(shape.num_experts, m_prime, 2).numpy()
    t0 = time.perf_counter()
    z = oracle.router_logits(x, wr)
    idx, gates = oracle.route(z, ret, shape.top_k)
    oracle.group_by_expert(idx, shape.num_experts)
    t_route = time.perf_counter() - t0
    se = None
    if layer.shared is not None:
        se = [t.cpu() for t in layer.shared]
        se = (se[0].numpy(), synth.bf16_bits(se[1]), synth.bf16_bits(se[2]))
    n, t_ffn = 0, 0.0
    while n < B and t_ffn < budget_s:
        t1 = time.perf_counter()
        o = oracle.experts_combine(x, idx, gates, gu, dn, tokens=[n])
        if se is not None:
            oracle.shared_expert_add(x, se[0], se[1], se[2], o, tokens=[n])
        t_ffn += time.perf_counter() - t1
        n += 1
    per_token = t_ffn / n + t_route / B
    return {"value": 1.0 / per_token, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"routing of all {B} tokens + expert FFNs/combine of {n} tokens of the "
                      f"{B}-token batch, single thread, {t_route + t_ffn:.1f} s of CPU work",
            "host_cpus": os.cpu_count()}


def weight_copies(wl, shape, sweep=False):
    """Weight copies a workload rotates through: one when the most expert bytes
    a step can touch exceed L2 several times, otherwise four."""
    B, m_prime = wl["B"], wl["m_prime"]
    most_touched = min(m_prime, B * shape.top_k) * shape.expert_bytes
    return 4 if (sweep or most_touched < 4 * L2_BYTES) else 1


def eq1_union(B, m_prime, k):
    """Expected distinct experts of a batch under uniform routing (Eq. 1)."""
    return m_prime * (1 - (1 - k / m_prime) ** B)


def workload_rotation(wl, shape):
    """Weight copies the GPU arm rotates across steps for this workload: four
    when the expected touched bytes (Eq. 1 union) stay under 4 x L2, else one."""
    touched = eq1_union(wl["B"], wl["m_prime"], shape.top_k) * shape.expert_bytes
    touched += 6 * shape.hidden * wl.get("shared", 0)
    copies = weight_copies(wl, shape)
    return copies if (copies > 1 and touched < 4 * L2_BYTES) else 1


def workload_config(name, wl, shape, ws):
    """The `config` object of a bench line.  It depends on the workload alone,
    so both arms print the same object; measured unions go in 'union'."""
    B, m_prime, k = wl["B"], wl["m_prime"], shape.top_k
    touched = eq1_union(B, m_prime, k) * shape.expert_bytes + 6 * shape.hidden * wl.get("shared", 0)
    l2 = ("touched expert weights about %.2f GB per step (Eq. 1 union) > 129 MB L2 (no flush needed)"
          % (touched / 1e9))
    rotated = workload_rotation(wl, shape)
    if rotated > 1:
        l2 += "; %d weight copies rotated across steps" % rotated
    return {"workload": name, "hidden": shape.hidden, "experts": shape.num_experts,
            "retained": m_prime, "inter": shape.inter, "top_k": k, "batch": B,
            "form": "compact checkpoint" if wl.get("compact") else "masked pool",
            "shared_expert_inter": wl.get("shared", 0),
            "parallelism": f"replicas{ws}", "l2": l2}


def main_gpu(args, ws, rank, local):
    import paper_2609_34117_gb300 as sw
    from paper_2609_34117_gb300 import build as swbuild
    if rank == 0 or ws == 1:
        swbuild.build()
    dist_barrier(ws)
    sw.load()
    device = torch.device("cuda", local)
    wl = WORKLOADS[args.workload]
    shape = SHAPES[wl.get("shape", "qwen")]
    B, m_prime = wl["B"], wl["m_prime"]
    # one weight copy is enough when the touched bytes exceed L2 several times;
    # otherwise (the sweep's small points, the most-pruned layers) 4 copies
    # rotate, as they do wherever the measured union stays under 4 x L2
    copies = weight_copies(wl, shape, args.sweep)
    layer = LayerInputs(shape, seed=0, device=device, copies=copies, shared=wl.get("shared", 0))
    sweep_layer = layer if layer.shared is None else LayerInputs(shape, 0, device, copies)
    full_shape = shape
    if wl.get("compact"):
        layer = layer.compacted(m_prime)
        shape = layer.shape
    torch.cuda.synchronize()
    torch.cuda.synchronize()
    peak, peak_kind = measured_peaks()

    with ClockSampler(local) as clk:
        dist_barrier(ws)
        pt = measure_point(sw, layer, B, m_prime, args.steps, args.warmup, device, seed_x=1,
                           soak_s=CLOCK_SOAK_S)
        dist_barrier(ws)
    tokens, secs = aggregate(ws, B * args.steps, pt["step_ms"] * 1e-3 * args.steps)
    value = tokens / secs
    graph = graph_measure(sw, layer, B, pt)
    e2e = e2e_measure(sw, layer, B, m_prime, min(args.steps, 2000), device, pt)
    e2e["value"] = e2e["value"] * ws  # replicas: all ranks' tokens
    achieved = pt["ffn_algo_bytes"] / (pt["ffn_ms"] * 1e-3) / 1e9
    result = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": pt["step_ms"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(args.workload, wl, full_shape, ws),
        "union": {"mean": pt["union_mean"], "eq1": pt["union_eq1"],
                  "weight_copies_rotated": pt["weight_copies_rotated"]},
        "touched_hbm": {"gbs": pt["touched_gbs"], "frac_of_8tbs": pt["touched_gbs"] / NOMINAL_HBM_GBS,
                        "frac_of_measured": pt["touched_gbs"] / peak},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "peak_kind": peak_kind,
                     "kernel": "expert_ffn_kernel", "kernel_ms": pt["ffn_ms"],
                     "algo_bytes_per_launch": pt["ffn_algo_bytes"],
                     "traffic": profiled_traffic(args.workload)},
        "e2e": e2e,
        "step_ms_p10_p50_p90": [pt["step_ms_p10"], pt["step_ms_p50"], pt["step_ms_p90"]],
        "step_spread": "percentiles of the mean step over blocks of 10 consecutive layer calls",
        "graph": graph,
        "gpu_launches": 4 * args.steps,   # route, group, expert FFN, combine per step
        "clocks": dict(clk.summary(), soak_s=CLOCK_SOAK_S),
    }
    if FFN_ITEMS:
        result["ffn_items"] = FFN_ITEMS
    if not args.no_pruned:
        result["pruned"] = run_pruned(sw, device, peak, local)
        result["compact_checkpoint"] = run_compact(sw, device, peak)
    if args.sweep:
        result["sweep"] = run_sweep(sw, sweep_layer, device, peak,
                                    cpu=rank == 0 and not args.no_cpu_baseline)
    if rank == 0 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(layer, B, m_prime)
    elif rank == 0:
        result["cpu_baseline"] = None
    if args.stack40:
        del layer
        torch.cuda.empty_cache()
        result["stack40"] = run_stack40(sw, device, max(3, min(args.steps // 100, 20)), 2, peak,
                                        cpu=rank == 0 and not args.no_cpu_baseline)
    if rank == 0:
        print(json.dumps(result), flush=True)


PRUNED_POINTS = ("qwen_p50_b64", "qwen_p50_b256", "qwen_p75_b64")

# form of the expert-FFN work items for the routed layers (--ffn-items; the
# C ABI's slimwise_decode_opts.ffn_items: 0 the default, 1 CTA-pair items)
FFN_ITEMS = 0

# untimed seconds of the headline layer's calls before its timed steps, inside
# the clock sampler's window (about 10 samples under load at any K)
CLOCK_SOAK_S = 1.0


def run_pruned(sw, device, peak, local, steps=4000):
    """The pruned Qwen-class layer at the target's points (50 % pruning at
    B = 64 and 256, 75 % at B = 64): each point times `steps` layer calls
    under its own clock sampler.  'touched' is the union's weight bytes over
    the whole step time (routing + grouping + FFN)."""
    shape = synth.QWEN
    layer = LayerInputs(shape, seed=0, device=device, copies=4)
    pts = []
    for name in PRUNED_POINTS:
        wl = WORKLOADS[name]
        with ClockSampler(local) as clk:
            p = measure_point(sw, layer, wl["B"], wl["m_prime"], steps, 50, device, seed_x=1)
        p.pop("_state")
        pts.append({
            "workload": name, "batch": wl["B"], "retained": wl["m_prime"], "steps": steps,
            "union_mean": p["union_mean"], "ms_per_step": p["step_ms"],
            "tokens_per_s": p["tokens_per_s"], "ffn_ms": p["ffn_ms"],
            "touched_gbs": p["touched_gbs"],
            "touched_frac_of_measured": p["touched_gbs"] / peak,
            "touched_frac_of_8tbs": p["touched_gbs"] / NOMINAL_HBM_GBS,
            "ffn_frac_of_measured": p["ffn_gbs"] / peak,
            "step_ms_p10_p50_p90": [p["step_ms_p10"], p["step_ms_p50"], p["step_ms_p90"]],
            "weight_copies_rotated": p["weight_copies_rotated"],
            "clocks": clk.summary()})
    del layer
    torch.cuda.empty_cache()
    return pts


def run_compact(sw, device, peak, m_prime=64, calls=50):
    """The compact checkpoint of the Qwen-class layer's m' = 64 retained experts
    (Sec. 3.1), built by slimwise_moe_compact_layer: model preparation, not a
    decode step.  Events around `calls` back-to-back calls (both launches of
    each); bytes = read + write of the retained experts' weights and router
    rows.  The result is checked against torch.index_select of the same rows."""
    shape = synth.QWEN
    w_gu, w_d = synth.expert_weights(shape, 0, device=device)
    wr = synth.router_weight(shape, 0, device=device)
    ret = synth.retained_set(shape.num_experts, m_prime, 2, shuffle=True).to(device)
    for _ in range(3):
        out = sw.slimwise_moe_compact_layer(w_gu, w_d, wr, ret)
    torch.cuda.synchronize()
    ids = torch.sort(ret.long()).values
    exact = (torch.equal(out[0], w_gu.index_select(0, ids)) and
             torch.equal(out[1], w_d.index_select(0, ids)) and
             torch.equal(out[2], wr.index_select(0, ids)) and torch.equal(out[3].long(), ids))
    del out
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(calls):
        sw.slimwise_moe_compact_layer(w_gu, w_d, wr, ret)
    b.record()
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / calls
    nbytes = 2 * m_prime * (shape.expert_bytes + shape.hidden * 4)
    del w_gu, w_d, wr
    torch.cuda.empty_cache()
    return {"retained": m_prime, "calls": calls, "ms": ms, "bytes": nbytes,
            "gbs": nbytes / (ms * 1e-3) / 1e9, "frac_of_measured": nbytes / (ms * 1e-3) / 1e9 / peak,
            "equals_index_select": bool(exact)}


def cpu_oracle_all_cores(w_gu_bits, w_d_bits, wr, retained, x_bits, k, tokens):
    """The oracle built with OpenMP over tokens, on all host cores: routing of
    the whole batch (single thread) and the expert FFNs + combine of `tokens`.
    Returns (seconds, threads) or None when no OpenMP build is possible."""
    import oracle
    try:
        path = oracle.build_openmp()
    except (OSError, subprocess.CalledProcessError):
        return None
    with oracle.swapped_library(path):
        threads = oracle.num_threads()
        t0 = time.perf_counter()
        idx, gates = oracle.route(oracle.router_logits(x_bits, wr), retained, k)
        oracle.group_by_expert(idx, wr.shape[0])
        oracle.experts_combine(x_bits, idx, gates, w_gu_bits, w_d_bits, tokens=tokens)
        return time.perf_counter() - t0, threads


def run_stack40(sw, device, steps, warmup, peak, n_layers=40, B=256, m_prime=64, cpu=False):
    """Decode-step MoE stack: n_layers independent Qwen-class layers (own
    weights, own retained set, own Zipf(1.1) popularity bias), called back to
    back on one stream; one step = all layers over one batch."""
    shape = synth.QWEN
    k = shape.top_k
    layers = []
    for l in range(n_layers):
        w_gu, w_d = synth.expert_weights(shape, 5000 + l, device=device)
        wr = synth.router_weight(shape, 5000 + l, device=device)
        bias = synth.zipf_rank_bias(shape.num_experts, 1.1, 9000 + l).to(device)
        wr[:, -1] = bias
        ret = synth.retained_set(shape.num_experts, m_prime, 7000 + l).to(device)
        layers.append((w_gu, w_d, wr, ret))
    x = synth.hidden_states(B, shape, 1, device=device)
    x[:, -1] = 1.0
    ws_buf = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, device)
    out = torch.empty((B, shape.hidden), dtype=torch.bfloat16, device=device)
    us = []
    for (w_gu, w_d, wr, ret) in layers:
        r = sw.slimwise_moe_route(x, wr, ret, k, shape.num_experts, shape.inter)
        us.append(int(r["union_size"].item()))
    stream = torch.cuda.current_stream()

    def one_step():
        for (w_gu, w_d, wr, ret) in layers:
            sw.slimwise_moe_decode_ex(x, wr, ret, w_gu, w_d, k, out=out, workspace=ws_buf, stream=stream)

    for _ in range(warmup):
        one_step()
    torch.cuda.synchronize()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(steps):
        one_step()
    t1.record(stream)
    torch.cuda.synchronize()
    if sw.slimwise_moe_device_status(ws_buf):
        raise RuntimeError("device error bits set in the stack run")
    ms = t0.elapsed_time(t1) / steps
    touched = sum(us) * shape.expert_bytes
    cpu_base = None
    if cpu:
        # the all-core oracle on the first 3 layers, whole batch each; the
        # stack's time is their mean per layer times the layer count
        xb = synth.bf16_bits(x)
        secs, threads = [], 1
        for (w_gu, w_d, wr, ret) in layers[:3]:
            r = cpu_oracle_all_cores(synth.bf16_bits(w_gu), synth.bf16_bits(w_d), wr.cpu().numpy(),
                                     ret.cpu().numpy(), xb, k, None)
            if r is None:
                break
            secs.append(r[0])
            threads = r[1]
        if secs:
            per_layer = float(np.mean(secs))
            cpu_base = {"value": B / (per_layer * n_layers), "unit": "tokens/s through the stack",
                        "cores": threads, "kind": "oracle (OpenMP over tokens)",
                        "sample": f"layers 0-2 of the {n_layers}, all {B} tokens each "
                                  f"({sum(secs):.1f} s); stack time = mean per layer x {n_layers}",
                        "host_cpus": os.cpu_count()}
    return {"layers": n_layers, "B": B, "m_prime": m_prime, "step_ms": ms,
            "cpu_baseline": cpu_base,
            "tokens_per_s_through_stack": B / (ms * 1e-3),
            "layer_tokens_per_s": B * n_layers / (ms * 1e-3),
            "union_per_layer": us, "union_mean": float(np.mean(us)),
            "touched_gb_per_step": touched / 1e9, "touched_gbs": touched / (ms * 1e-3) / 1e9,
            "touched_frac_of_measured": touched / (ms * 1e-3) / 1e9 / peak,
            "weights_gb": n_layers * shape.num_experts * shape.expert_bytes / 1e9}


def run_sweep(sw, layer, device, peak, cpu=False):
    gu_bits = dn_bits = wr = None
    if cpu:
        w_gu, w_d = layer.copies[0]
        gu_bits, dn_bits, wr = synth.bf16_bits(w_gu), synth.bf16_bits(w_d), layer.wr.cpu().numpy()
    shape = layer.shape
    pts = []
    for B in (1, 8, 32, 64, 128, 256, 512):
        for m_prime in (128, 96, 64, 32):
            steps = 300 if B <= 64 else 200
            p = measure_point(sw, layer, B, m_prime, steps, 20, device, seed_x=1000 + B)
            batches, retained = p.pop("_state")[:2]
            p["touched_frac_of_measured"] = p["touched_gbs"] / peak
            p["ffn_frac_of_measured"] = p["ffn_gbs"] / peak
            if cpu:
                # the all-core oracle on the point's first batch, every token
                ret = None if retained is None else retained.cpu().numpy()
                r = cpu_oracle_all_cores(gu_bits, dn_bits, wr, ret, synth.bf16_bits(batches[0]),
                                         shape.top_k, None)
                p["cpu_baseline"] = None if r is None else {
                    "value": B / r[0], "unit": "tokens/s", "cores": r[1],
                    "kind": "oracle (OpenMP over tokens)", "sample": f"one batch of {B} tokens",
                    "host_cpus": os.cpu_count()}
            pts.append(p)
    return pts


# ---------------------------------------------------------------- reference arm
def main_reference(args, ws, rank):
    """The reference arm is the CPU oracle, timed as it stands on one host core.

    Each step is the layer over one batch: routing of all B tokens, then the
    expert FFNs and combine of the batch's tokens -- all of them when the
    whole --steps/--warmup run fits in about two minutes at the oracle's
    speed, else the first n tokens that fit.  ms_per_step is the measured wall
    time of a step; value = tokens processed / wall time."""
    if rank != 0:
        return
    import oracle
    oracle.build()
    wl = WORKLOADS[args.workload]
    shape = SHAPES[wl.get("shape", "qwen")]
    B, m_prime = wl["B"], wl["m_prime"]
    w_gu, w_d = synth.expert_weights(shape, 0)
    wr = synth.router_weight(shape, 0).numpy()
    gu, dn = synth.bf16_bits(w_gu), synth.bf16_bits(w_d)
    ret = None if m_prime >= shape.num_experts else synth.retained_set(shape.num_experts, m_prime, 2).numpy()
    se = None
    if wl.get("shared"):
        w_sg, gu_s, dn_s = synth.shared_expert(shape.hidden, wl["shared"], 0 + 101)
        se = (w_sg.numpy(), synth.bf16_bits(gu_s), synth.bf16_bits(dn_s))
    full_shape = shape
    if wl.get("compact"):
        # the retained experts' rows only, in ascending id order
        gu, dn, wr, _ = oracle.compact_layer(gu, dn, wr, ret)
        shape = synth.LayerShape(shape.hidden, m_prime, shape.inter, shape.top_k)
        ret = None
    batches = [synth.bf16_bits(synth.hidden_states(B, shape, 1 + j)) for j in range(N_BATCHES)]
    # the union of each batch, as the GPU arm reports it
    unions = [oracle.group_by_expert(oracle.route(oracle.router_logits(xb, wr), ret, shape.top_k)[0],
                                     shape.num_experts)["union_size"] for xb in batches]

    def step(i, n_tok):
        x = batches[i % N_BATCHES]
        t0 = time.perf_counter()
        z = oracle.router_logits(x, wr)
        idx, gates = oracle.route(z, ret, shape.top_k)
        oracle.group_by_expert(idx, shape.num_experts)
        toks = list(range(n_tok))
        o = oracle.experts_combine(x, idx, gates, gu, dn, tokens=toks)
        if se is not None:
            oracle.shared_expert_add(x, se[0], se[1], se[2], o, tokens=toks)
        return time.perf_counter() - t0

    # size the step from one timed token so the whole run stays bounded
    per_tok = step(0, 1)
    budget_s = 120.0
    n_tok = int(max(1, min(B, budget_s / (args.steps + args.warmup) / max(per_tok, 1e-6))))
    for i in range(args.warmup):
        step(i, n_tok)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(i, n_tok)
    wall = time.perf_counter() - t0
    ms = wall / args.steps * 1e3
    value = n_tok * args.steps / wall
    sample = (f"per step: routing of all {B} tokens, expert FFNs + combine of "
              + (f"all {B} tokens" if n_tok == B else f"the first {n_tok} of {B} tokens")
              + ", single thread")
    print(json.dumps({
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
        "config": workload_config(args.workload, wl, full_shape, ws),
        "union": {"mean": float(np.mean(unions)), "eq1": eq1_union(B, m_prime, full_shape.top_k)},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": sample, "host_cpus": os.cpu_count()},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=4000)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", default="slimwise", choices=["slimwise", "reference"])
    ap.add_argument("--workload", default="qwen_full_b64", choices=sorted(WORKLOADS))
    ap.add_argument("--sweep", action="store_true", help="batch x pruning sweep (adds 'sweep')")
    ap.add_argument("--stack40", action="store_true",
                    help="40 independent skewed layers at m'=64, B=256 (adds 'stack40')")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--ffn-items", type=int, default=0, choices=[-1, 0, 1],
                    help="expert-FFN work items: 0 default, 1 CTA-pair items")
    ap.add_argument("--no-pruned", action="store_true",
                    help="skip the pruned-layer points (adds 'pruned' by default)")
    args = ap.parse_args()
    global FFN_ITEMS
    FFN_ITEMS = args.ffn_items
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    ws, rank, local = dist_init()
    if args.impl == "reference":
        main_reference(args, ws, rank)
    else:
        main_gpu(args, ws, rank, local)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
