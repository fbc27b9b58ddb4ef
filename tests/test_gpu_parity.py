"""Parity of the CUDA decode MoE layer (through the C ABI) with the CPU oracle.

Integer results -- top-k ids, union, counts, offsets, grouped permutation --
must match bit for bit.  Outputs (bf16 in, fp32 accumulate, bf16 out) must be
within relative L2 error 1e-2 and max-abs error 3e-2 of the oracle's fp64
values; gates within fp32 rounding of the oracle's.  At the Qwen-class sizes
the routing of every token is checked and outputs on a seeded sample of
tokens the oracle evaluates one by one.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2609_34117_gb300 as sw
from paper_2609_34117_gb300 import synth

pytestmark = pytest.mark.gpu

REL_L2_TOL = 1e-2
MAX_ABS_TOL = 3e-2
GATE_RTOL = 4e-6
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    sw.build.build()
    oracle.build()


class Layer:
    def __init__(self, shape, seed=0):
        self.shape = shape
        self.w_gu, self.w_d = synth.expert_weights(shape, seed)
        self.wr = synth.router_weight(shape, seed)
        self.gu_bits = synth.bf16_bits(self.w_gu)
        self.d_bits = synth.bf16_bits(self.w_d)
        self.d_w_gu = self.w_gu.to(DEV)
        self.d_w_d = self.w_d.to(DEV)
        self.d_wr = self.wr.to(DEV)


@pytest.fixture(scope="module")
def tiny():
    return Layer(synth.TINY, seed=0)


@pytest.fixture(scope="module")
def qwen():
    return Layer(synth.QWEN, seed=0)


@pytest.fixture(scope="module")
def qwen36():
    return Layer(synth.QWEN36, seed=0)


def _run(layer, x, retained, k, wr=None, workspace=None):
    wr_d = layer.d_wr if wr is None else wr.to(DEV)
    xd = x.to(DEV)
    if retained is None:
        out = sw.slimwise_moe_decode_full(xd, wr_d, layer.d_w_gu, layer.d_w_d, k, workspace=workspace)
    else:
        out = sw.slimwise_moe_decode(xd, wr_d, retained.to(DEV), layer.d_w_gu, layer.d_w_d, k,
                                     workspace=workspace)
    route = sw.slimwise_moe_route(xd, wr_d, None if retained is None else retained.to(DEV), k,
                                  layer.shape.num_experts, layer.shape.inter)
    torch.cuda.synchronize()
    return out, {n: t.cpu().numpy() for n, t in route.items()}


def _oracle(layer, x, retained, k, tokens=None, wr=None):
    wr_np = (layer.wr if wr is None else wr).numpy()
    ret = None if retained is None else retained.numpy()
    xb = synth.bf16_bits(x)
    if tokens is None:
        r = oracle.moe_decode(xb, wr_np, ret, layer.gu_bits, layer.d_bits, k)
    else:
        r = oracle.moe_decode_sampled(xb, wr_np, ret, layer.gu_bits, layer.d_bits, k, tokens)
    r["group"] = oracle.group_by_expert(r["idx"], layer.shape.num_experts)
    return r


def _check_route(route, ref, E):
    assert np.array_equal(route["topk_idx"], ref["idx"])
    np.testing.assert_allclose(route["topk_gate"], ref["gates"], rtol=GATE_RTOL, atol=1e-7)
    g = ref["group"]
    assert np.array_equal(route["counts"], g["counts"])
    assert np.array_equal(route["offsets"], g["offsets"])
    assert int(route["union_size"][0]) == g["union_size"]
    U = g["union_size"]
    assert np.array_equal(route["union_ids"][:U], g["union_ids"])
    assert np.all(route["union_ids"][U:] == -1)
    assert np.array_equal(route["perm"], g["perm"])
    assert np.array_equal(route["pos"], g["pos"])


def _check_out(got, ref):
    got = got.astype(np.float64)
    err = np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30)
    mx = float(np.abs(got - ref).max()) if ref.size else 0.0
    assert err <= REL_L2_TOL and mx <= MAX_ABS_TOL, (err, mx)
    return err, mx


def _case(layer, B, m_prime, seed_x, seed_imp, k=None, sample=None, shuffle=False, x=None, wr=None):
    shape = layer.shape
    k = shape.top_k if k is None else k
    if x is None:
        x = synth.hidden_states(B, shape, seed_x)
    retained = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, seed_imp,
                                                                shuffle=shuffle)
    out, route = _run(layer, x, retained, k, wr=wr)
    tokens = None
    if sample is not None and B > sample:
        tokens = np.sort(np.random.default_rng(seed_x).choice(B, size=sample, replace=False)).astype(np.int32)
    ref = _oracle(layer, x, retained, k, tokens=tokens, wr=wr)
    _check_route(route, ref, shape.num_experts)
    got = out.float().cpu().numpy()
    if tokens is not None:
        got = got[tokens]
    return _check_out(got, ref["out"]), out, route


# --------------------------------------------------------------------------
def test_tiny_layer_matches_oracle(tiny):
    (err, mx), _, _ = _case(tiny, B=4, m_prime=8, seed_x=1, seed_imp=2)
    assert err < 5e-3


def test_closed_form_golden_layer():
    from tests.golden.closed_form import B, E, H, I, build_case
    case = build_case()
    with open(os.path.join(os.path.dirname(__file__), "golden", "closed_form_layer.json")) as f:
        gold = json.load(f)
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a)).view(dt).to(DEV)  # noqa: E731
    x = t(case["x"].view(np.int16), torch.bfloat16)
    gu = t(case["w_gate_up"].view(np.int16), torch.bfloat16).view(E, 2 * I, H)
    dn = t(case["w_down"].view(np.int16), torch.bfloat16).view(E, H, I)
    wr = torch.from_numpy(case["router_w"]).to(DEV)
    ret = torch.from_numpy(case["retained"]).to(DEV)
    out = sw.slimwise_moe_decode(x.view(B, H), wr, ret, gu, dn, case["k"])
    route = sw.slimwise_moe_route(x.view(B, H), wr, ret, case["k"], E, I)
    torch.cuda.synchronize()
    assert route["topk_idx"].cpu().tolist() == gold["idx"]
    np.testing.assert_allclose(route["topk_gate"].cpu().numpy(), np.array(gold["gates"]), rtol=GATE_RTOL)
    _check_out(out.float().cpu().numpy(), np.array(gold["out"]))


def test_qwen_full_pool_b64(qwen):
    # the headline layer: every output of the batch against the oracle
    _case(qwen, B=64, m_prime=None, seed_x=1, seed_imp=2)


@pytest.mark.parametrize("B", [64, 128, 256])
def test_qwen_pruned_50pct(qwen, B):
    # every output at B = 64, 32 sampled tokens above
    _case(qwen, B=B, m_prime=64, seed_x=1, seed_imp=2, sample=None if B == 64 else 32)


@pytest.mark.parametrize("B,m_prime", [(1, 128), (8, 96), (32, 32), (128, 96), (512, 32), (512, 128)])
def test_qwen_sweep_points(qwen, B, m_prime):
    _case(qwen, B=B, m_prime=m_prime, seed_x=1000 + B, seed_imp=2 + m_prime, sample=32)


@pytest.mark.parametrize("B", [31, 33, 65, 151, 153, 303, 305, 319])
@pytest.mark.parametrize("m_prime", [None, 32])
def test_routing_at_cluster_size_boundaries(qwen, B, m_prime):
    # Routing clusters take 1, 2, 4, 8 or 16 tokens as B grows (thresholds
    # 32, 64, 152, 304), staged in token pairs from 2 tokens on and summed
    # two tokens at a time with packed multiply-adds.  Batches just either
    # side of each threshold end a cluster on an odd token, so the last pair
    # holds one real token beside a zero row: every token's top-k ids and
    # gates, the union and the grouping must still equal the oracle's bit for
    # bit (routing only; the layer's outputs are covered by the other cases).
    shape = qwen.shape
    x = synth.hidden_states(B, shape, 2000 + B)
    retained = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, 9)
    route = sw.slimwise_moe_route(x.to(DEV), qwen.d_wr, None if retained is None else retained.to(DEV),
                                  shape.top_k, shape.num_experts, shape.inter)
    torch.cuda.synchronize()
    idx, gates = oracle.route(oracle.router_logits(synth.bf16_bits(x), qwen.wr.numpy()),
                              None if retained is None else retained.numpy(), shape.top_k)
    ref = {"idx": idx, "gates": gates, "group": oracle.group_by_expert(idx, shape.num_experts)}
    _check_route({n: t.cpu().numpy() for n, t in route.items()}, ref, shape.num_experts)


@pytest.mark.parametrize("B,m_prime", [(64, 192), (64, 128), (256, 64), (8, 64)])
def test_qwen36_shaped_layer(qwen36, B, m_prime):
    # 256 experts of intermediate size 512: 25 / 50 / 75 % pruning
    _case(qwen36, B=B, m_prime=m_prime, seed_x=3000 + B, seed_imp=2 + m_prime, sample=16)


@pytest.mark.parametrize("m_prime", [64, 32])
def test_compact_checkpoint_equals_masked_pool(qwen, m_prime):
    # Sec. 3.1: the Eq. 2 mask over the full pool and a checkpoint holding only
    # the retained experts give the same layer
    from paper_2609_34117_gb300 import checkpoint
    shape = qwen.shape
    retained = synth.retained_set(shape.num_experts, m_prime, 5, shuffle=True).to(DEV)
    gu_c, d_c, wr_c, ids = checkpoint.compact_layer(qwen.d_w_gu, qwen.d_w_d, qwen.d_wr, retained)
    assert gu_c.numel() * shape.num_experts == qwen.d_w_gu.numel() * m_prime
    x = synth.hidden_states(96, shape, 21).to(DEV)
    masked = sw.slimwise_moe_decode(x, qwen.d_wr, retained, qwen.d_w_gu, qwen.d_w_d, 8)
    compact = sw.slimwise_moe_decode_full(x, wr_c, gu_c, d_c, 8)
    r_m = sw.slimwise_moe_route(x, qwen.d_wr, retained, 8, shape.num_experts, shape.inter)
    r_c = sw.slimwise_moe_route(x, wr_c, None, 8, m_prime, shape.inter)
    torch.cuda.synchronize()
    assert torch.equal(masked, compact)
    ids_d = ids.to(DEV).long()
    assert torch.equal(ids_d[r_c["topk_idx"].long()], r_m["topk_idx"].long())
    assert torch.equal(r_c["topk_gate"], r_m["topk_gate"])
    assert torch.equal(r_c["perm"], r_m["perm"])
    assert torch.equal(r_c["counts"], r_m["counts"][ids_d])
    assert int(r_c["union_size"][0]) == int(r_m["union_size"][0])
    # the compact form against the oracle run on the compact tensors (expert
    # ids in compact numbering), every token's routing, 32 tokens' outputs
    xb = synth.bf16_bits(x)
    tokens = np.sort(np.random.default_rng(m_prime).choice(96, size=32, replace=False)).astype(np.int32)
    ref = oracle.moe_decode_sampled(xb, wr_c.cpu().numpy(), None, synth.bf16_bits(gu_c),
                                    synth.bf16_bits(d_c), 8, tokens)
    ref["group"] = oracle.group_by_expert(ref["idx"], m_prime)
    _check_route({n: t.cpu().numpy() for n, t in r_c.items()}, ref, m_prime)
    _check_out(compact.float().cpu().numpy()[tokens], ref["out"])
    # and mapped back to original ids it is the masked pool's routing
    ref_m = oracle.route(oracle.router_logits(xb, qwen.wr.numpy()), retained.cpu().numpy(), 8)
    assert np.array_equal(ids.cpu().numpy()[ref["idx"]], ref_m[0])


@pytest.mark.parametrize("shape_name,m_prime", [("tiny", 8), ("tiny", 16), ("qwen", 64), ("qwen", 1)])
def test_compact_layer_kernel_equals_oracle_compaction(request, shape_name, m_prime):
    # The compaction kernels (slimwise_moe_compact_layer) against the oracle's
    # compaction of the same host tensors: every byte of the compact weights
    # and router rows, and the ids, in ascending original order (a shuffled
    # retained list; all experts, reversed; one expert).
    layer = request.getfixturevalue(shape_name)
    E = layer.shape.num_experts
    if m_prime == E:
        retained = torch.arange(E - 1, -1, -1, dtype=torch.int32)
    else:
        retained = synth.retained_set(E, m_prime, 7, shuffle=True)
    gu_c, d_c, wr_c, ids = sw.slimwise_moe_compact_layer(layer.d_w_gu, layer.d_w_d, layer.d_wr,
                                                         retained.to(DEV))
    torch.cuda.synchronize()
    r_gu, r_d, r_wr, r_ids = oracle.compact_layer(layer.gu_bits, layer.d_bits, layer.wr.numpy(),
                                                  retained.numpy())
    assert np.array_equal(ids.cpu().numpy(), r_ids)
    assert np.array_equal(synth.bf16_bits(gu_c.cpu()), r_gu)
    assert np.array_equal(synth.bf16_bits(d_c.cpu()), r_d)
    assert np.array_equal(wr_c.cpu().numpy().view(np.uint32), r_wr.view(np.uint32))


def test_compact_layer_kernel_rejects_repeated_and_out_of_range_ids(tiny):
    from paper_2609_34117_gb300 import checkpoint
    E = tiny.shape.num_experts
    for bad in ([3, 5, 3, 9], [0, E, 2], [-1, 4]):
        ret = torch.tensor(bad, dtype=torch.int32, device=DEV)
        gu_c, d_c, wr_c, ids = sw.slimwise_moe_compact_layer(tiny.d_w_gu, tiny.d_w_d, tiny.d_wr, ret)
        torch.cuda.synchronize()
        assert bool((ids == -1).all())
        with pytest.raises(ValueError):
            checkpoint.compact_layer(tiny.d_w_gu, tiny.d_w_d, tiny.d_wr, ret)
    # and a good call on the same stream afterwards is unaffected
    ret = synth.retained_set(E, 8, 3).to(DEV)
    _, _, _, ids = sw.slimwise_moe_compact_layer(tiny.d_w_gu, tiny.d_w_d, tiny.d_wr, ret)
    assert torch.equal(ids, torch.sort(ret).values)


class SharedExpert:
    def __init__(self, layer, inter_shared, seed):
        H = layer.shape.hidden
        self.w_sg, self.gu, self.dn = synth.shared_expert(H, inter_shared, seed)
        self.gu_bits, self.dn_bits = synth.bf16_bits(self.gu), synth.bf16_bits(self.dn)
        self.d_w_sg, self.d_gu, self.d_dn = self.w_sg.to(DEV), self.gu.to(DEV), self.dn.to(DEV)


def _case_shared(layer, se, B, m_prime, seed_x, seed_imp, k=None, sample=None, x=None):
    shape = layer.shape
    k = shape.top_k if k is None else k
    if x is None:
        x = synth.hidden_states(B, shape, seed_x)
    retained = None if m_prime is None else synth.retained_set(shape.num_experts, m_prime, seed_imp)
    out = sw.slimwise_moe_decode_shared(x.to(DEV), layer.d_wr, None if retained is None else retained.to(DEV),
                                        layer.d_w_gu, layer.d_w_d, k, se.d_w_sg, se.d_gu, se.d_dn)
    torch.cuda.synchronize()
    tokens = None
    if sample is not None and B > sample:
        tokens = np.sort(np.random.default_rng(seed_x).choice(B, size=sample, replace=False)).astype(np.int32)
    ref = oracle.moe_decode_shared(synth.bf16_bits(x), layer.wr.numpy(),
                                   None if retained is None else retained.numpy(), layer.gu_bits,
                                   layer.d_bits, k, se.w_sg.numpy(), se.gu_bits, se.dn_bits, tokens)
    got = out.float().cpu().numpy()
    if tokens is not None:
        got = got[tokens]
    return _check_out(got, ref["out"]), out


@pytest.fixture(scope="module")
def tiny_shared(tiny):
    return SharedExpert(tiny, 128, seed=31)


@pytest.fixture(scope="module")
def qwen36_shared(qwen36):
    # Sec. 3.3: the distilled decoder's shared expert is twice the original width
    return SharedExpert(qwen36, 1024, seed=32)


@pytest.mark.parametrize("B", [1, 4, 17, 300])
def test_shared_expert_layer_tiny(tiny, tiny_shared, B):
    # B = 300 spans two shared-expert work entries of 256 tokens
    _case_shared(tiny, tiny_shared, B=B, m_prime=8, seed_x=40 + B, seed_imp=2)


@pytest.mark.parametrize("B,m_prime", [(64, 128), (256, 64)])
def test_shared_expert_layer_qwen36(qwen36, qwen36_shared, B, m_prime):
    _case_shared(qwen36, qwen36_shared, B=B, m_prime=m_prime, seed_x=50 + B, seed_imp=2 + m_prime,
                 sample=6)


def test_shared_expert_closed_gate_is_the_routed_layer(tiny, tiny_shared):
    # gate logit -1000 for every token: s_t = 0 and the output is exactly the
    # routed layer's
    shape = tiny.shape
    x = synth.hidden_states(24, shape, 61)
    x[:, -1] = 1.0
    w_sg = torch.zeros(shape.hidden, dtype=torch.float32)
    w_sg[-1] = -1000.0
    retained = synth.retained_set(shape.num_experts, 8, 2).to(DEV)
    xd = x.to(DEV)
    with_se = sw.slimwise_moe_decode_shared(xd, tiny.d_wr, retained, tiny.d_w_gu, tiny.d_w_d, 2,
                                            w_sg.to(DEV), tiny_shared.d_gu, tiny_shared.d_dn)
    routed = sw.slimwise_moe_decode(xd, tiny.d_wr, retained, tiny.d_w_gu, tiny.d_w_d, 2)
    torch.cuda.synchronize()
    assert torch.equal(with_se, routed)


@pytest.mark.parametrize("B,m_prime,hot", [(128, None, 1), (200, None, 2), (256, 8, 1)])
def test_hot_expert_spans_several_slots(B, m_prime, hot):
    # One or two experts chosen by every token, the rest of the load spread
    # thin: the token chunk follows the mean load (16 or 128 rows), so a hot
    # expert becomes several work entries, each streaming the expert's weight
    # tiles for its own chunk of tokens.  (256, 8): 64 tokens per retained
    # expert on average, three entries for the hot one.
    shape = synth.LayerShape(hidden=256, num_experts=64, inter=128, top_k=2)
    layer = Layer(shape, seed=11)
    retained = None if m_prime is None else synth.retained_set(64, m_prime, 13)
    hot_ids = [5, 17] if retained is None else [int(retained[2])]
    bias = torch.zeros(64)
    for j, e in enumerate(hot_ids[:hot]):
        bias[e] = 8.0 - 2.0 * j
    x, wr = synth.apply_popularity_bias(synth.hidden_states(B, shape, 140 + B), layer.wr, bias)
    _, _, route = _case(layer, B=B, m_prime=m_prime, seed_x=140 + B, seed_imp=13, x=x, wr=wr)
    assert route["counts"].max() == B


@pytest.mark.parametrize("B,skew", [(256, False), (256, True), (200, False)])
def test_wide_items_every_output(B, skew):
    # 64 of 128 experts, top-8: a mean load of 32 (25 at B = 200) gives token
    # chunks of 64 rows, where each work item covers two adjacent 128-row
    # weight tiles sharing each stage's token rows (two accumulators per
    # item).  Every output and the whole routing against the oracle, with
    # uniform and Zipf-skewed routing (popular experts in several entries).
    shape = synth.LayerShape(hidden=256, num_experts=128, inter=256, top_k=8)
    layer = Layer(shape, seed=19)
    x, wr = synth.hidden_states(B, shape, 160 + B), None
    if skew:
        bias = synth.zipf_rank_bias(shape.num_experts, 1.1, 161)
        x, wr = synth.apply_popularity_bias(x, layer.wr, bias)
    _case(layer, B=B, m_prime=64, seed_x=160 + B, seed_imp=21, x=x, wr=wr)


@pytest.mark.parametrize("B", [1, 5, 17, 33, 300])
def test_ragged_batches_and_token_chunks(tiny, B):
    # k = m' = 8: every token selects every retained expert, so each expert
    # holds B tokens and B = 300 exceeds one 256-token work item
    _case(tiny, B=B, m_prime=8, seed_x=B, seed_imp=2, k=8)


@pytest.mark.parametrize("k", [1, 2, 8])
def test_top_k_extremes(tiny, k):
    _case(tiny, B=12, m_prime=8, seed_x=7, seed_imp=3, k=k)


@pytest.mark.parametrize("B,k", [(33, 12), (300, 16)])
def test_top_k_above_8(tiny, B, k):
    # the full tiny pool (16 experts) with k > 8: every combine sums two
    # batches of selections; at B = 300 most experts hold two work entries
    _case(tiny, B=B, m_prime=None, seed_x=50 + k, seed_imp=0, k=k)


def test_top_k_32_qwen(qwen):
    # the largest k the ABI accepts, on the Qwen-class full pool
    _case(qwen, B=8, m_prime=None, seed_x=61, seed_imp=0, k=32, sample=4)


@pytest.mark.parametrize("B", [37, 200])
def test_generic_shape(B):
    # H = 640 (five 128-wide chunks: ragged batches of router-row loads, five
    # combine tiles), I = 192 (three gate/up tiles), 24 experts, top-3 of 12;
    # B = 200 gives token chunks of 80 rows (not a power of two)
    layer = Layer(synth.LayerShape(hidden=640, num_experts=24, inter=192, top_k=3), seed=3)
    _case(layer, B=B, m_prime=12, seed_x=70 + B, seed_imp=4)


@pytest.mark.parametrize("B", [5, 90])
def test_generic_shape_with_shared_expert(B):
    # the generic shape with a shared expert of width 192 (three gate/up
    # tiles, three down K stages); B = 90 makes two shared entries of 64
    layer = Layer(synth.LayerShape(hidden=640, num_experts=24, inter=192, top_k=3), seed=3)
    se = SharedExpert(layer, 192, seed=33)
    _case_shared(layer, se, B=B, m_prime=12, seed_x=80 + B, seed_imp=4)


@pytest.mark.parametrize("B", [200, 400])
def test_wide_hidden(B):
    # H = 8192: 8 or 16 tokens per routing cluster would stage more hidden
    # rows than a CTA's shared memory holds, so the clusters take fewer tokens
    layer = Layer(synth.LayerShape(hidden=8192, num_experts=64, inter=128, top_k=4), seed=5)
    _case(layer, B=B, m_prime=32, seed_x=90 + B, seed_imp=6, sample=4)


@pytest.mark.parametrize("E,m_prime,k,B", [(512, 384, 8, 40), (1024, 1024, 32, 4)])
def test_large_pools(E, m_prime, k, B):
    # more than 256 retained experts: the routing's general top-k (candidates
    # in a local array), up to the largest pool and k the ABI accepts
    layer = Layer(synth.LayerShape(hidden=256, num_experts=E, inter=64, top_k=k), seed=7)
    _case(layer, B=B, m_prime=None if m_prime == E else m_prime, seed_x=95 + B, seed_imp=8)


def test_wide_intermediate():
    # I = 4096: 64 gate/up tiles per entry and 64 K stages per down item
    layer = Layer(synth.LayerShape(hidden=256, num_experts=8, inter=4096, top_k=2), seed=9)
    _case(layer, B=10, m_prime=6, seed_x=97, seed_imp=10)


def test_zero_tokens_is_noop(tiny):
    x = torch.empty((0, tiny.shape.hidden), dtype=torch.bfloat16, device=DEV)
    out = sw.slimwise_moe_decode_full(x, tiny.d_wr, tiny.d_w_gu, tiny.d_w_d, 2)
    torch.cuda.synchronize()
    assert out.shape == (0, tiny.shape.hidden)


def test_retained_order_irrelevant_and_full_equals_all(qwen):
    shape = qwen.shape
    x = synth.hidden_states(64, shape, 11).to(DEV)
    r_sorted = synth.retained_set(shape.num_experts, 64, 2).to(DEV)
    r_shuf = synth.retained_set(shape.num_experts, 64, 2, shuffle=True).to(DEV)
    a = sw.slimwise_moe_decode(x, qwen.d_wr, r_sorted, qwen.d_w_gu, qwen.d_w_d, 8)
    b = sw.slimwise_moe_decode(x, qwen.d_wr, r_shuf, qwen.d_w_gu, qwen.d_w_d, 8)
    full = sw.slimwise_moe_decode_full(x, qwen.d_wr, qwen.d_w_gu, qwen.d_w_d, 8)
    allr = torch.arange(shape.num_experts, dtype=torch.int32, device=DEV).flip(0).contiguous()
    c = sw.slimwise_moe_decode(x, qwen.d_wr, allr, qwen.d_w_gu, qwen.d_w_d, 8)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert torch.equal(full, c)


def test_batch_permutation_and_determinism(qwen):
    shape = qwen.shape
    x = synth.hidden_states(96, shape, 12).to(DEV)
    ret = synth.retained_set(shape.num_experts, 64, 2).to(DEV)
    a = sw.slimwise_moe_decode(x, qwen.d_wr, ret, qwen.d_w_gu, qwen.d_w_d, 8)
    a2 = sw.slimwise_moe_decode(x, qwen.d_wr, ret, qwen.d_w_gu, qwen.d_w_d, 8)
    p = torch.randperm(96, generator=torch.Generator().manual_seed(0)).to(DEV)
    b = sw.slimwise_moe_decode(x[p].contiguous(), qwen.d_wr, ret, qwen.d_w_gu, qwen.d_w_d, 8)
    torch.cuda.synchronize()
    assert torch.equal(a, a2)
    diff = (a[p].float() - b.float()).abs().max().item()
    assert diff <= 1e-2 * a.float().abs().max().item()


def test_workspace_contents_do_not_matter(tiny):
    shape = tiny.shape
    x = synth.hidden_states(9, shape, 4).to(DEV)
    ret = synth.retained_set(shape.num_experts, 8, 2).to(DEV)
    ws = sw.alloc_workspace(9, shape.hidden, shape.num_experts, shape.inter, 2, DEV)
    ws.fill_(0xFF)
    a = sw.slimwise_moe_decode(x, tiny.d_wr, ret, tiny.d_w_gu, tiny.d_w_d, 2, workspace=ws)
    ws.fill_(0x00)
    b = sw.slimwise_moe_decode(x, tiny.d_wr, ret, tiny.d_w_gu, tiny.d_w_d, 2, workspace=ws)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert sw.slimwise_moe_device_status(ws) == 0


@pytest.mark.parametrize("fill", [0xFF, 0x00])
def test_long_combine_lists_all_outputs(tiny, fill):
    # 600 tokens, k = 4 of m' = 8: 300 tokens per retained expert, two work
    # entries each, and 2,400 (token, h tile) combines; a workspace of 0xFF
    # or 0x00 bytes must not change anything
    shape = tiny.shape
    B, k = 600, 4
    x = synth.hidden_states(B, shape, 21)
    retained = synth.retained_set(shape.num_experts, 8, 5)
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, DEV)
    ws.fill_(fill)
    out = sw.slimwise_moe_decode(x.to(DEV), tiny.d_wr, retained.to(DEV), tiny.d_w_gu, tiny.d_w_d,
                                 k, workspace=ws)
    torch.cuda.synchronize()
    assert sw.slimwise_moe_device_status(ws) == 0
    ref = _oracle(tiny, x, retained, k)
    _check_out(out.float().cpu().numpy(), ref["out"])


@pytest.mark.parametrize("B", [127, 128])
def test_combine_grid_ragged_and_full(tiny, B):
    # k = 2 of m' = 8: B * H/128 (token, tile) combines, one per warp of the
    # combine kernel's 8-warp CTAs -- a ragged last CTA at B = 127, full CTAs
    # at B = 128.  Every output against the oracle.
    _case(tiny, B=B, m_prime=8, seed_x=31 + B, seed_imp=6, k=2)


def test_duplicate_retained_id_is_reported(tiny):
    shape = tiny.shape
    x = synth.hidden_states(4, shape, 4).to(DEV)
    ret = torch.tensor([1, 3, 3, 7, 9], dtype=torch.int32, device=DEV)
    ws = sw.alloc_workspace(4, shape.hidden, shape.num_experts, shape.inter, 2, DEV)
    sw.slimwise_moe_decode(x, tiny.d_wr, ret, tiny.d_w_gu, tiny.d_w_d, 2, workspace=ws)
    assert sw.slimwise_moe_device_status(ws) & sw.binding.DEVERR_DUPLICATE_RETAINED
    ok = torch.tensor([1, 3, 7, 9], dtype=torch.int32, device=DEV)
    sw.slimwise_moe_decode(x, tiny.d_wr, ok, tiny.d_w_gu, tiny.d_w_d, 2, workspace=ws)
    assert sw.slimwise_moe_device_status(ws) == 0


def test_top1_one_hot_router_is_dense_ffn(tiny):
    shape = tiny.shape
    ret = synth.retained_set(shape.num_experts, 8, 2)
    e_star = int(ret[5])
    x, wr = synth.apply_popularity_bias(synth.hidden_states(16, shape, 5), tiny.wr, torch.zeros(shape.num_experts))
    wr[e_star, -1] = 8.0
    out, route = _run(tiny, x, ret, 1, wr=wr)
    assert np.all(route["topk_idx"][:, 0] == e_star)
    assert np.all(route["topk_gate"] == 1.0)
    x64 = x.double().numpy()
    gu = tiny.w_gu[e_star].double().numpy()
    dn = tiny.w_d[e_star].double().numpy()
    I = shape.inter
    g, u = x64 @ gu[:I].T, x64 @ gu[I:].T
    ref = (g / (1 + np.exp(-g)) * u) @ dn.T
    _check_out(out.float().cpu().numpy(), ref)


def test_group_of_uniform_selections_matches_oracle_and_eq1():
    E, k, m_prime, B, draws = 128, 8, 64, 16, 200
    rng = np.random.default_rng(9)
    pool = np.sort(rng.choice(E, size=m_prime, replace=False))
    us = []
    for _ in range(draws):
        sel = np.stack([rng.choice(pool, size=k, replace=False) for _ in range(B)]).astype(np.int32)
        g = sw.slimwise_moe_group(torch.from_numpy(sel).to(DEV), E, hidden=2048, inter=768)
        ref = oracle.group_by_expert(sel, E)
        U = int(g["union_size"].item())
        assert U == ref["union_size"]
        assert np.array_equal(g["perm"].cpu().numpy(), ref["perm"])
        assert np.array_equal(g["offsets"].cpu().numpy(), ref["offsets"])
        us.append(U)
    us = np.array(us, np.float64)
    expect = m_prime * (1 - (1 - k / m_prime) ** B)
    assert abs(us.mean() - expect) <= 4 * us.std(ddof=1) / math.sqrt(draws) + 1e-9


def test_zipf_skewed_layers_route_exactly(qwen):
    shape = qwen.shape
    B, m_prime = 256, 64
    x0 = synth.hidden_states(B, shape, 77)
    ret = synth.retained_set(shape.num_experts, m_prime, 2)
    for layer_seed in (0, 1):
        bias = synth.zipf_rank_bias(shape.num_experts, 1.1, 100 + layer_seed)
        x, wr = synth.apply_popularity_bias(x0, qwen.wr, bias)
        _case(qwen, B=B, m_prime=m_prime, seed_x=5, seed_imp=2, sample=4, x=x, wr=wr)
    # skew concentrates tokens, so at a small batch fewer distinct experts are
    # touched than Eq. 1 predicts for uniform routing (Sec. 2.1)
    Bs, us = 16, []
    for layer_seed in range(4):
        bias = synth.zipf_rank_bias(shape.num_experts, 1.1, 200 + layer_seed)
        x, wr = synth.apply_popularity_bias(synth.hidden_states(Bs, shape, 300 + layer_seed), qwen.wr, bias)
        r = sw.slimwise_moe_route(x.to(DEV), wr.to(DEV), ret.to(DEV), 8, shape.num_experts, shape.inter)
        us.append(int(r["union_size"].item()))
    assert np.mean(us) < m_prime * (1 - (1 - 8 / m_prime) ** Bs)


def test_layer_stack_40_layers_back_to_back():
    # The decode-step MoE stack the benchmark times: 40 distinct Qwen-class
    # layers (own weights, retained set and Zipf(1.1) popularity; 48 GB of
    # expert weights drawn on the device with the benchmark's seeds) run back
    # to back through one workspace.  Every layer's routing, union and
    # grouping is checked exactly against the oracle; the outputs of layers
    # 0, 19 and 39 on 16 sampled tokens (their weights copied to the host).
    shape = synth.QWEN
    B, m_prime, k, n_layers = 256, 64, shape.top_k, 40
    x = synth.hidden_states(B, shape, 1, device=DEV)
    x[:, -1] = 1.0
    ws = sw.alloc_workspace(B, shape.hidden, shape.num_experts, shape.inter, k, DEV)
    layers, outs = [], []
    for l in range(n_layers):
        w_gu, w_d = synth.expert_weights(shape, 5000 + l, device=DEV)
        wr = synth.router_weight(shape, 5000 + l, device=DEV)
        wr[:, -1] = synth.zipf_rank_bias(shape.num_experts, 1.1, 9000 + l).to(DEV)
        ret = synth.retained_set(shape.num_experts, m_prime, 7000 + l).to(DEV)
        layers.append((w_gu, w_d, wr, ret))
    for (w_gu, w_d, wr, ret) in layers:
        outs.append(sw.slimwise_moe_decode(x, wr, ret, w_gu, w_d, k, workspace=ws))
    torch.cuda.synchronize()
    assert sw.slimwise_moe_device_status(ws) == 0
    xb = synth.bf16_bits(x)
    tokens = np.sort(np.random.default_rng(3).choice(B, size=16, replace=False)).astype(np.int32)
    unions = []
    for l, (w_gu, w_d, wr, ret) in enumerate(layers):
        route = sw.slimwise_moe_route(x, wr, ret, k, shape.num_experts, shape.inter)
        route = {n: t.cpu().numpy() for n, t in route.items()}
        wr_h, ret_h = wr.cpu().numpy(), ret.cpu().numpy()
        if l in (0, 19, 39):
            ref = oracle.moe_decode_sampled(xb, wr_h, ret_h, synth.bf16_bits(w_gu), synth.bf16_bits(w_d),
                                            k, tokens)
            _check_out(outs[l].float().cpu().numpy()[tokens], ref["out"])
        else:
            idx, gates = oracle.route(oracle.router_logits(xb, wr_h), ret_h, k)
            ref = {"idx": idx, "gates": gates}
        ref["group"] = oracle.group_by_expert(ref["idx"], shape.num_experts)
        _check_route(route, ref, shape.num_experts)
        unions.append(ref["group"]["union_size"])
    # skewed popularity still touches most of a 64-expert pool at B = 256
    assert min(unions) >= 32 and max(unions) <= m_prime


# --------------------------------------------------------------------------
# Expert-importance statistics and the retained set (Sec. 2.3, Sec. 3.1)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("layer_name,B,k", [("tiny", 40, 2), ("qwen", 64, 8)])
def test_expert_stats_match_oracle(request, layer_name, B, k):
    layer = request.getfixturevalue(layer_name)
    shape = layer.shape
    stats = None
    ref = np.zeros((shape.num_experts, 4))
    for batch in range(2):   # statistics accumulate over calibration batches
        x = synth.hidden_states(B, shape, 70 + batch)
        stats, out = sw.slimwise_moe_expert_stats(x.to(DEV), layer.d_wr, layer.d_w_gu, layer.d_w_d, k,
                                                  stats=stats)
        ref = oracle.expert_stats(synth.bf16_bits(x), layer.wr.numpy(), layer.gu_bits, layer.d_bits, k,
                                  stats=ref)
        # the calibration pass's layer output is the full-pool layer
        full = sw.slimwise_moe_decode_full(x.to(DEV), layer.d_wr, layer.d_w_gu, layer.d_w_d, k)
        torch.cuda.synchronize()
        assert torch.equal(out, full)
    got = stats.cpu().numpy()
    assert np.array_equal(got[:, 0], ref[:, 0])                      # tokens routed: exact
    np.testing.assert_allclose(got[:, 1], ref[:, 1], rtol=1e-5, atol=1e-6)   # fp32 gates
    # norms of fp32 expert outputs computed through a bf16 activation
    np.testing.assert_allclose(got[:, 2], ref[:, 2], rtol=1e-2, atol=1e-6)
    np.testing.assert_allclose(got[:, 3], ref[:, 3], rtol=1e-2, atol=1e-6)
    # the device selection is the oracle's selection of the same statistics
    for crit in ("mass", "ean", "reap"):
        for m in (1, shape.num_experts // 2, shape.num_experts):
            ids = sw.slimwise_moe_select_retained(stats, m, crit).cpu().numpy()
            assert np.array_equal(ids, oracle.select_retained(got, m, crit)), (crit, m)


def test_select_retained_ties_and_extremes():
    E = 100
    rng = np.random.default_rng(5)
    st = np.zeros((E, 4))
    st[:, 0] = rng.integers(0, 3, E)
    st[:, 1] = rng.integers(0, 4, E) * 0.25
    st[:, 2] = rng.integers(0, 4, E) * 0.5
    st[:, 3] = st[:, 1] * st[:, 2]
    d = torch.from_numpy(st).to(DEV)
    for crit in ("mass", "ean", "reap"):
        for m in (0, 1, 37, E):
            ids = sw.slimwise_moe_select_retained(d, m, crit).cpu().numpy()
            assert np.array_equal(ids, oracle.select_retained(st, m, crit)), (crit, m)
    # all scores equal: the lowest ids
    z = torch.zeros((E, 4), dtype=torch.float64, device=DEV)
    assert np.array_equal(sw.slimwise_moe_select_retained(z, 10, "reap").cpu().numpy(), np.arange(10))
