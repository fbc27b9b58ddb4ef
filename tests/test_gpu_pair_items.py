"""CTA-pair work items of the expert FFN against the CPU oracle.

A pair item puts an item's two 128-row weight tiles on the two CTAs of a
cluster, which run one M = 256 tcgen05 MMA whose token rows are split between
their shared memories.  The launch option ffn_items = 1 selects them; here
on layers of every size, so that ragged batches, single tokens, several
entries per expert, skewed routing, the largest token chunk and the timeout
path all run through the pair form.  The bar is the
one of every other parity test: routing exact, outputs within rel-L2 1e-2
and max-abs 3e-2 of the oracle's fp64 values.
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
REL_L2_TOL = 1e-2
MAX_ABS_TOL = 3e-2


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()
    oracle.build()


class _Layer:
    def __init__(self, shape, seed):
        self.shape = shape
        self.w_gu, self.w_d = synth.expert_weights(shape, seed)
        self.wr = synth.router_weight(shape, seed)
        self.d_w_gu, self.d_w_d = self.w_gu.to(DEV), self.w_d.to(DEV)


_LAYERS = {}


def _layer(name):
    if name not in _LAYERS:
        shapes = {
            "tiny": (synth.TINY, 0),
            # H 256, 128 experts of I 256, top-8: many items per entry
            "mid": (synth.LayerShape(hidden=256, num_experts=128, inter=256, top_k=8), 19),
        }
        shape, seed = shapes[name]
        _LAYERS[name] = _Layer(shape, seed)
    return _LAYERS[name]


def _decode(layer, x, wr, retained, k, ffn_items, workspace=None, **kw):
    return sw.slimwise_moe_decode_ex(x.to(DEV), wr.to(DEV),
                                     None if retained is None else retained.to(DEV),
                                     layer.d_w_gu, layer.d_w_d, k, workspace=workspace,
                                     ffn_items=ffn_items, **kw)


def _oracle(layer, x, wr, retained, k, tokens=None):
    args = (synth.bf16_bits(x), wr.numpy(), None if retained is None else retained.numpy(),
            synth.bf16_bits(layer.w_gu), synth.bf16_bits(layer.w_d), k)
    if tokens is None:
        return oracle.moe_decode(*args)
    return oracle.moe_decode_sampled(*args, tokens)


def _check_out(got, ref):
    got = got.astype(np.float64)
    err = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    mx = float(np.abs(got - ref).max()) if ref.size else 0.0
    assert err <= REL_L2_TOL and mx <= MAX_ABS_TOL, (err, mx)
    return err, mx


def _pair_case(name, B, m_prime, seed, skew=False, k=None):
    layer = _layer(name)
    shape = layer.shape
    k = shape.top_k if k is None else k
    x, wr = synth.hidden_states(B, shape, seed), layer.wr
    if skew:
        x, wr = synth.apply_popularity_bias(x, wr, synth.zipf_rank_bias(shape.num_experts, 1.1,
                                                                        seed + 1))
    retained = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, seed + 2)
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, DEV)
    out = _decode(layer, x, wr, retained, k, ffn_items=1, workspace=ws)
    flags = sw.slimwise_moe_device_status(ws)
    assert flags == 0, flags
    ref = _oracle(layer, x, wr, retained, k)
    err, mx = _check_out(out.float().cpu().numpy(), ref["out"])
    return layer, x, wr, retained, k, out, ws


# one token, ragged batches, several entries per expert (B = 600, skewed
# routing); token chunks from 16 to 112 rows, and 224 (B = 512 over 24
# experts: all 512 TMEM columns)
@pytest.mark.parametrize("name,B,m_prime,skew", [
    ("tiny", 4, 8, False), ("tiny", 33, 8, False), ("mid", 1, 64, False),
    ("mid", 17, None, False), ("mid", 64, 64, False), ("mid", 200, 64, False),
    ("mid", 256, 64, True), ("mid", 600, 64, False), ("mid", 600, 64, True),
    ("mid", 512, 24, False)])
def test_pair_items_every_output(name, B, m_prime, skew):
    _pair_case(name, B, m_prime, seed=700 + B, skew=skew)


def test_pair_items_equal_single_cta_items():
    # the same layer through pair items and through 128-row items: both within
    # the tolerance of the oracle, and close to each other
    layer, x, wr, retained, k, out_pair, ws = _pair_case("mid", 200, 32, seed=811)
    out_one = _decode(layer, x, wr, retained, k, ffn_items=-1, workspace=ws)
    torch.cuda.synchronize()
    d = (out_pair.float() - out_one.float()).abs().max().item()
    assert d <= 1e-2, d


@pytest.mark.parametrize("B,m_prime", [(512, 32), (300, 32)])
def test_pair_items_qwen_class(B, m_prime):
    # the Qwen-class layer at large token chunks (176 and 112 rows), where
    # pair items would halve the token rows each SM reads; outputs of 32
    # sampled tokens
    shape = synth.QWEN
    key = "qwen"
    if key not in _LAYERS:
        _LAYERS[key] = _Layer(shape, 0)
    layer = _LAYERS[key]
    x = synth.hidden_states(B, shape, 5000 + B)
    retained = synth.retained_set(shape.num_experts, m_prime, 2 + m_prime)
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, shape.top_k, DEV)
    out = _decode(layer, x, layer.wr, retained, shape.top_k, ffn_items=1, workspace=ws)
    assert sw.slimwise_moe_device_status(ws) == 0
    tokens = np.sort(np.random.default_rng(B).choice(B, size=32, replace=False)).astype(np.int32)
    ref = _oracle(layer, x, layer.wr, retained, shape.top_k, tokens=tokens)
    _check_out(out.float().cpu().numpy()[tokens], ref["out"])


@pytest.mark.parametrize("B", [8, 300])
def test_pair_items_dependency_wait_runs_out(B):
    # the timeout path with pair items: the first routed down item waits for a
    # gate/up tile that never exists; both CTAs of its pair give up after the
    # short limit, the call reports it, and the next call is clean
    layer = _layer("tiny")
    shape = layer.shape
    k = shape.top_k
    x = synth.hidden_states(B, shape, 90 + B)
    retained = synth.retained_set(shape.num_experts, 8, 2)
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, DEV)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    _decode(layer, x, layer.wr, retained, k, ffn_items=1, workspace=ws, wait_limit_ns=2_000_000,
            test_starve_first_down=True)
    flags = sw.slimwise_moe_device_status(ws)
    elapsed = time.perf_counter() - t0
    assert flags & sw.binding.DEVERR_DEPENDENCY_TIMEOUT, flags
    assert not flags & sw.binding.DEVERR_TMEM_PAIR, flags
    assert elapsed < 0.5, elapsed
    out = _decode(layer, x, layer.wr, retained, k, ffn_items=1, workspace=ws)
    assert sw.slimwise_moe_device_status(ws) == 0
    ref = _oracle(layer, x, layer.wr, retained, k)
    _check_out(out.float().cpu().numpy(), ref["out"])
