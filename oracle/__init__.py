"""CPU oracle for the SlimWise pruned-pool batched-decode MoE layer.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg are the only callers.  The CUDA product
path never imports this package, and this package imports nothing from the
product.

The arithmetic lives in ``slimwise_oracle.c`` (plain C loops, fp32 routing in
the canonical order, fp64 everything after the routing decision); this module
only compiles it with gcc and marshals numpy arrays through ctypes.  Each
wrapper names the paper passage its C function follows.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "slimwise_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_OMP_PATH = os.path.join(_BUILD_DIR, "liboracle_omp.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FP contraction)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
           "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def build_openmp(force: bool = False) -> str:
    """The same source built with -fopenmp: the tokens of the expert/combine
    step run on all host cores.  Used only to time the oracle on all cores."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_OMP_PATH)
            and os.path.getmtime(_OMP_PATH) >= os.path.getmtime(_SRC)):
        return _OMP_PATH
    tmp = _OMP_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC",
           "-shared", "-std=c11", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True, capture_output=True)
    os.replace(tmp, _OMP_PATH)
    return _OMP_PATH


def num_threads() -> int:
    """Threads the loaded library's token loop uses (1 for the plain build)."""
    return int(_load().oracle_num_threads())


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32 = ctypes.c_int
            lib.oracle_router_logits.argtypes = [P, P, i32, i32, i32, P]
            lib.oracle_router_logits.restype = None
            lib.oracle_route.argtypes = [P, i32, i32, P, i32, i32, P, P]
            lib.oracle_route.restype = i32
            lib.oracle_group_by_expert.argtypes = [P, i32, i32, i32, P, P, P, P, P, P]
            lib.oracle_group_by_expert.restype = None
            lib.oracle_expert_swiglu.argtypes = [P, P, P, i32, i32, P, P]
            lib.oracle_expert_swiglu.restype = None
            lib.oracle_experts_combine.argtypes = [P, P, P, P, P, i32, i32, i32, P, i32, P]
            lib.oracle_experts_combine.restype = i32
            lib.oracle_shared_expert_add.argtypes = [P, P, P, P, i32, i32, P, i32, P, P]
            lib.oracle_shared_expert_add.restype = i32
            lib.oracle_expert_stats.argtypes = [P, P, P, P, i32, i32, i32, i32, i32, P]
            lib.oracle_expert_stats.restype = i32
            lib.oracle_select_retained.argtypes = [P, i32, i32, i32, P]
            lib.oracle_select_retained.restype = i32
            lib.oracle_moe_decode.argtypes = [P, P, P, i32, P, P, i32, i32, i32, i32, i32, P, P, P]
            lib.oracle_moe_decode.restype = i32
            lib.oracle_num_threads.argtypes = []
            lib.oracle_num_threads.restype = i32
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _c(a, dtype):
    a = np.ascontiguousarray(a)
    if a.dtype != dtype:
        raise TypeError(f"expected {dtype}, got {a.dtype}")
    return a


def router_logits(x_bf16: np.ndarray, router_w: np.ndarray) -> np.ndarray:
    """Router logits z = x Wr^T in the canonical fp32 order (Sec. 3.1).

    x_bf16: uint16 [B, H] (bf16 bit patterns); router_w: fp32 [E, H].
    Returns fp32 [B, E].
    """
    x = _c(x_bf16, np.uint16)
    w = _c(router_w, np.float32)
    B, H = x.shape
    E = w.shape[0]
    if H % 128:
        raise ValueError("H must be a multiple of 128")
    z = np.empty((B, E), np.float32)
    _load().oracle_router_logits(_ptr(x), _ptr(w), B, H, E, _ptr(z))
    return z


def route(z: np.ndarray, retained, k: int):
    """Eq. 2 masking, top-k and renormalised gates (Sec. 3.1).

    retained: int32 ids of K' (any order) or None for the full pool.
    Returns (idx int32 [B, k], gates fp64 [B, k]).
    """
    z = _c(z, np.float32)
    B, E = z.shape
    r = None if retained is None else _c(np.asarray(retained, np.int32), np.int32)
    idx = np.empty((B, k), np.int32)
    gates = np.empty((B, k), np.float64)
    rc = _load().oracle_route(_ptr(z), B, E, _ptr(r), 0 if r is None else len(r),
                              k, _ptr(idx), _ptr(gates))
    if rc != 0:
        raise ValueError("oracle_route: bad arguments")
    return idx, gates


def group_by_expert(idx: np.ndarray, E: int) -> dict:
    """Counts, offsets, union and grouped permutation of the routed slots (Eq. 1)."""
    idx = _c(idx, np.int32)
    B, k = idx.shape
    counts = np.empty(E, np.int32)
    offsets = np.empty(E + 1, np.int32)
    union_ids = np.empty(E, np.int32)
    usize = np.zeros(1, np.int32)
    perm = np.empty(B * k, np.int32)
    pos = np.empty(B * k, np.int32)
    _load().oracle_group_by_expert(_ptr(idx), B, k, E, _ptr(counts), _ptr(offsets),
                                   _ptr(union_ids), _ptr(usize), _ptr(perm), _ptr(pos))
    u = int(usize[0])
    return {"counts": counts, "offsets": offsets, "union_ids": union_ids[:u].copy(),
            "union_size": u, "perm": perm, "pos": pos}


def expert_swiglu(x_row: np.ndarray, w_gate_up_e: np.ndarray, w_down_e: np.ndarray):
    """One expert on one token: SwiGLU in fp64. Returns (act [I], y [H])."""
    x = _c(x_row, np.uint16)
    wgu = _c(w_gate_up_e, np.uint16)
    wd = _c(w_down_e, np.uint16)
    H = x.shape[0]
    I = wgu.shape[0] // 2
    a = np.empty(I, np.float64)
    y = np.empty(H, np.float64)
    _load().oracle_expert_swiglu(_ptr(x), _ptr(wgu), _ptr(wd), H, I, _ptr(a), _ptr(y))
    return a, y


def experts_combine(x_bf16, idx, gates, w_gate_up, w_down, tokens=None):
    """Expert FFNs + gate-weighted combine for `tokens` (default: all). fp64 [n, H]."""
    x = _c(x_bf16, np.uint16)
    idx = _c(idx, np.int32)
    gates = _c(gates, np.float64)
    wgu = _c(w_gate_up, np.uint16)
    wd = _c(w_down, np.uint16)
    B, H = x.shape
    k = idx.shape[1]
    I = wgu.shape[1] // 2
    toks = np.arange(B, dtype=np.int32) if tokens is None else _c(np.asarray(tokens, np.int32), np.int32)
    out = np.empty((len(toks), H), np.float64)
    rc = _load().oracle_experts_combine(_ptr(x), _ptr(idx), _ptr(gates), _ptr(wgu), _ptr(wd),
                                        H, I, k, _ptr(toks), len(toks), _ptr(out))
    if rc != 0:
        raise MemoryError("oracle_experts_combine")
    return out


def shared_expert_add(x_bf16, w_shared_gate, w_shared_gu, w_shared_down, out, tokens=None):
    """Sec. 3.3 shared expert: adds s_t * SE(x_t) to `out` (fp64 [n, H], one row per
    token of `tokens`) in place; returns the gates s_t (fp64 [n])."""
    x = _c(x_bf16, np.uint16)
    wsg = _c(np.asarray(w_shared_gate, np.float32).reshape(-1), np.float32)
    gu = _c(w_shared_gu, np.uint16)
    wd = _c(w_shared_down, np.uint16)
    B, H = x.shape
    I_s = gu.shape[0] // 2
    toks = np.arange(B, dtype=np.int32) if tokens is None else _c(np.asarray(tokens, np.int32), np.int32)
    assert out.dtype == np.float64 and out.flags.c_contiguous and out.shape == (len(toks), H)
    s = np.empty(len(toks), np.float64)
    rc = _load().oracle_shared_expert_add(_ptr(x), _ptr(wsg), _ptr(gu), _ptr(wd), H, I_s,
                                          _ptr(toks), len(toks), _ptr(out), _ptr(s))
    if rc != 0:
        raise MemoryError("oracle_shared_expert_add")
    return s


CRITERIA = {"mass": 0, "ean": 1, "reap": 2}


def expert_stats(x_bf16, router_w, w_gate_up, w_down, k, stats=None):
    """Sec. 2.3 importance statistics of one calibration batch, full pool:
    fp64 [E, 4] = (tokens routed, routing mass, EAN, REAP numerator), added
    to `stats` when given."""
    x = _c(x_bf16, np.uint16)
    w = _c(router_w, np.float32)
    wgu = _c(w_gate_up, np.uint16)
    wd = _c(w_down, np.uint16)
    B, H = x.shape
    E = w.shape[0]
    I = wgu.shape[1] // 2
    if stats is None:
        stats = np.zeros((E, 4), np.float64)
    assert stats.dtype == np.float64 and stats.shape == (E, 4) and stats.flags.c_contiguous
    rc = _load().oracle_expert_stats(_ptr(x), _ptr(w), _ptr(wgu), _ptr(wd), B, H, E, I, k, _ptr(stats))
    if rc != 0:
        raise ValueError("oracle_expert_stats")
    return stats


def select_retained(stats, m_prime, criterion):
    """Top-m' experts by `criterion` ('mass', 'ean' or 'reap'), ties to the
    lowest id; int32 ids ascending."""
    st = _c(stats, np.float64)
    E = st.shape[0]
    ids = np.empty(m_prime, np.int32)
    if _load().oracle_select_retained(_ptr(st), E, int(m_prime), CRITERIA[criterion], _ptr(ids)) != 0:
        raise ValueError("oracle_select_retained: bad arguments")
    return ids


def moe_decode(x_bf16, router_w, retained, w_gate_up, w_down, k):
    """Whole decode layer over the retained pool (retained=None: full pool).

    Returns dict(idx int32 [B,k], gates fp64 [B,k], out fp64 [B,H]).
    """
    x = _c(x_bf16, np.uint16)
    w = _c(router_w, np.float32)
    wgu = _c(w_gate_up, np.uint16)
    wd = _c(w_down, np.uint16)
    B, H = x.shape
    E = w.shape[0]
    I = wgu.shape[1] // 2
    r = None if retained is None else _c(np.asarray(retained, np.int32), np.int32)
    idx = np.empty((B, k), np.int32)
    gates = np.empty((B, k), np.float64)
    out = np.empty((B, H), np.float64)
    rc = _load().oracle_moe_decode(_ptr(x), _ptr(w), _ptr(r), 0 if r is None else len(r),
                                   _ptr(wgu), _ptr(wd), B, H, E, I, k,
                                   _ptr(idx), _ptr(gates), _ptr(out))
    if rc != 0:
        raise ValueError("oracle_moe_decode: bad arguments")
    return {"idx": idx, "gates": gates, "out": out}


def moe_decode_sampled(x_bf16, router_w, retained, w_gate_up, w_down, k, tokens):
    """Routing for every token, expert FFN + combine only for `tokens`.

    Routing is per token, so the sampled rows equal the rows of the full layer.
    Returns dict(idx, gates, out [len(tokens), H], z).
    """
    z = router_logits(x_bf16, router_w)
    idx, gates = route(z, retained, k)
    out = experts_combine(x_bf16, idx, gates, w_gate_up, w_down, tokens)
    return {"idx": idx, "gates": gates, "out": out, "z": z}


def moe_decode_shared(x_bf16, router_w, retained, w_gate_up, w_down, k, w_shared_gate,
                      w_shared_gu, w_shared_down, tokens=None):
    """The layer with its shared expert (Sec. 3.3): routed experts as in
    `moe_decode`, then s_t * SE(x_t) added.  Expert FFNs for `tokens` only
    (default: all).  Returns dict(idx, gates, shared_gate, out)."""
    z = router_logits(x_bf16, router_w)
    idx, gates = route(z, retained, k)
    out = experts_combine(x_bf16, idx, gates, w_gate_up, w_down, tokens)
    s = shared_expert_add(x_bf16, w_shared_gate, w_shared_gu, w_shared_down, out, tokens)
    return {"idx": idx, "gates": gates, "shared_gate": s, "out": out}


def compact_layer(w_gate_up: np.ndarray, w_down: np.ndarray, router_w: np.ndarray, retained):
    """The pruned checkpoint of one layer (Sec. 3.1): the weights and router
    rows of the retained experts K' only, in ascending original id, so that
    top-k ties in the compact numbering still go to the lowest original id.

    Returns (w_gate_up_c [m', 2I, H], w_down_c [m', H, I], router_w_c [m', H],
    ids int32 [m']); compact expert j is original expert ids[j].  Raises on a
    repeated or out-of-range id.
    """
    ids = np.sort(np.asarray(retained, np.int64).ravel())
    E = w_gate_up.shape[0]
    if ids.size == 0 or ids[0] < 0 or ids[-1] >= E or np.any(ids[1:] == ids[:-1]):
        raise ValueError("retained ids must be distinct and in [0, E)")
    return (np.ascontiguousarray(w_gate_up[ids]), np.ascontiguousarray(w_down[ids]),
            np.ascontiguousarray(router_w[ids]), ids.astype(np.int32))


# ---------------------------------------------------------------------------
# Mutation support for the pin suite: compile a modified copy of the oracle
# source and swap it in, so a test can check that the pins catch a planted
# mistake.  Used only by tests.
# ---------------------------------------------------------------------------
def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def build_variant(src_text: str, tag: str) -> str:
    os.makedirs(_BUILD_DIR, exist_ok=True)
    src = os.path.join(_BUILD_DIR, f"variant_{tag}.c")
    out = os.path.join(_BUILD_DIR, f"variant_{tag}.so")
    with open(src, "w") as f:
        f.write(src_text)
    subprocess.run(["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
                    "-std=c11", "-o", out, src, "-lm"], check=True)
    return out


class swapped_library:
    """Context manager: route every wrapper through the library at `path`."""

    def __init__(self, path: str):
        self.path = path
        self.saved = None

    def __enter__(self):
        global _lib
        base = _load()
        lib = ctypes.CDLL(self.path)
        for name in ("oracle_router_logits", "oracle_route", "oracle_group_by_expert",
                     "oracle_expert_swiglu", "oracle_experts_combine", "oracle_moe_decode",
                     "oracle_shared_expert_add", "oracle_expert_stats", "oracle_select_retained",
                     "oracle_num_threads"):
            fn_new, fn_old = getattr(lib, name), getattr(base, name)
            fn_new.argtypes, fn_new.restype = fn_old.argtypes, fn_old.restype
        with _lock:
            self.saved, _lib = base, lib
        return lib

    def __exit__(self, *exc):
        global _lib
        with _lock:
            _lib = self.saved
        return False
