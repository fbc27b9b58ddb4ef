"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: a summation
error bound, brute-force enumeration, a closed form, an equivalence stated in
Sec. 3.1, an invariant, or the exact expectation of Eq. 1.  A plausible slip in
the oracle (a dropped term, a wrong sign, index or transpose) fails one of them.
"""
import itertools
import math

import numpy as np
import pytest
import torch

from paper_2609_34117_gb300 import synth

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


def _bits(t):
    return synth.bf16_bits(t)


def _bf16_to_f64(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _tiny_layer(seed=0, B=4, shape=synth.TINY):
    w_gu, w_d = synth.expert_weights(shape, seed)
    wr = synth.router_weight(shape, seed)
    x = synth.hidden_states(B, shape, seed + 1)
    return x, wr, w_gu, w_d


# --------------------------------------------------------------------------
# Router logits (Sec. 3.1): canonical fp32 sum vs exact dot product
# --------------------------------------------------------------------------
def test_logits_within_summation_error_bound(oracle_lib):
    x, wr, _, _ = _tiny_layer(B=6)
    xb = _bits(x)
    w = wr.numpy()
    z = oracle_lib.router_logits(xb, w)
    x64 = _bf16_to_f64(xb)
    w64 = w.astype(np.float64)
    exact = x64 @ w64.T
    absdot = np.abs(x64) @ np.abs(w64).T
    H = x64.shape[1]
    n_ops = H // 32 + 5          # depth of the canonical summation tree
    u = 2.0 ** -24
    gamma = n_ops * u / (1 - n_ops * u)
    err = np.abs(z.astype(np.float64) - exact)
    assert np.all(err <= gamma * absdot), float((err / (gamma * absdot + 1e-300)).max())
    # the bound is far below a typical single product, so dropping or
    # misplacing one term of the dot product would violate it
    typical = np.median(np.abs(x64[:, None, :] * w64[None, :, :]))
    assert gamma * absdot.max() < 0.01 * typical


def test_logits_exact_on_representable_inputs(oracle_lib):
    # x one-hot-ish with small integers and Wr with dyadic values: every product
    # and partial sum is exact, so the canonical order must give the exact value.
    rng = np.random.default_rng(1)
    B, H, E = 3, 256, 5
    xv = rng.integers(-4, 5, size=(B, H)).astype(np.float32)
    wv = (rng.integers(-64, 65, size=(E, H)) / 64.0).astype(np.float32)
    xb = torch.from_numpy(xv).to(torch.bfloat16)
    z = oracle_lib.router_logits(_bits(xb), wv)
    np.testing.assert_array_equal(z.astype(np.float64), xv.astype(np.float64) @ wv.astype(np.float64).T)


# --------------------------------------------------------------------------
# Top-k with lowest-id tie-break: brute force over all k-subsets
# --------------------------------------------------------------------------
def _brute_topk(zrow, retained, k):
    cand = sorted(retained)
    best = None
    for sub in itertools.combinations(cand, k):
        rest = [e for e in cand if e not in sub]
        # every chosen expert must beat every other retained expert on
        # (logit desc, id asc); IEEE comparison, so -0 == +0
        ok = all((zrow[a] > zrow[b]) or (zrow[a] == zrow[b] and a < b) for a in sub for b in rest)
        if ok:
            assert best is None, "two subsets satisfy the top-k condition"
            best = sub
    assert best is not None
    return sorted(best, key=lambda e: (-float(zrow[e]), e))


@pytest.mark.parametrize("seed", range(6))
def test_topk_matches_brute_force_with_ties(oracle_lib, seed):
    rng = np.random.default_rng(seed)
    B, E = 7, 9
    # few distinct values -> many ties; include signed zeros
    vals = np.array([-1.5, -0.0, 0.0, 0.5, 0.5, 2.0], np.float32)
    z = vals[rng.integers(0, len(vals), size=(B, E))].astype(np.float32)
    m_prime = int(rng.integers(3, E + 1))
    retained = rng.choice(E, size=m_prime, replace=False).astype(np.int32)
    for k in range(1, m_prime + 1):
        idx, gates = oracle_lib.route(z, retained, k)
        for t in range(B):
            assert list(idx[t]) == _brute_topk(z[t], retained.tolist(), k)


def test_zero_router_selects_lowest_retained_ids_with_equal_gates(oracle_lib):
    x, _, _, _ = _tiny_layer()
    E, H = synth.TINY.num_experts, synth.TINY.hidden
    wr = np.zeros((E, H), np.float32)
    z = oracle_lib.router_logits(_bits(x), wr)
    assert np.all(z == 0)
    retained = np.array([11, 3, 7, 14, 5, 9, 0, 12], np.int32)
    for k in (1, 2, 4, 8):
        idx, gates = oracle_lib.route(z, retained, k)
        assert np.all(idx == np.sort(retained)[:k])
        assert np.all(gates == 1.0 / k)   # exact for powers of two


# --------------------------------------------------------------------------
# Gates: renormalisation over the selected k (Sec. 3.1)
# --------------------------------------------------------------------------
def test_gates_equal_pool_softmax_renormalised_over_topk(oracle_lib):
    rng = np.random.default_rng(3)
    B, E, k = 16, 32, 4
    z = (rng.standard_normal((B, E)) * 3).astype(np.float32)
    retained = np.sort(rng.choice(E, size=20, replace=False)).astype(np.int32)
    idx, gates = oracle_lib.route(z, retained, k)
    zr = z[:, retained].astype(np.float64)
    p = np.exp(zr - zr.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)                        # softmax over the retained pool
    full = np.zeros((B, E))
    full[:, retained] = p
    sel = np.take_along_axis(full, idx, 1)
    ref = sel / sel.sum(1, keepdims=True)               # renormalise over the k selected
    np.testing.assert_allclose(gates, ref, rtol=1e-12, atol=0)
    np.testing.assert_allclose(gates.sum(1), 1.0, rtol=0, atol=k * 2.0 ** -52)
    assert np.all(np.diff(gates, axis=1) <= 0)          # selection order = gate order


def test_gates_independent_of_removed_unselected_experts(oracle_lib):
    rng = np.random.default_rng(4)
    B, E, k = 8, 24, 3
    z = rng.standard_normal((B, E)).astype(np.float32)
    retained = np.arange(E, dtype=np.int32)
    idx, gates = oracle_lib.route(z, retained, k)
    for t in range(B):
        chosen = set(idx[t].tolist())
        # drop every retained expert that token t did not select, except one
        keep = np.array(sorted(chosen | {next(e for e in range(E) if e not in chosen)}), np.int32)
        i2, g2 = oracle_lib.route(z[t:t + 1], keep, k)
        assert list(i2[0]) == list(idx[t])
        assert np.array_equal(g2[0], gates[t])


# --------------------------------------------------------------------------
# Masked router == pruned checkpoint (Sec. 3.1, Eq. 2); full pool == unpruned
# --------------------------------------------------------------------------
def test_masked_router_equals_pruned_checkpoint(oracle_lib):
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=5)
    retained = synth.retained_set(shape.num_experts, 8, seed=2, shuffle=True).numpy()
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    a = oracle_lib.moe_decode(xb, w, retained, gu, dn, shape.top_k)
    # pruned checkpoint: only the retained experts and their router rows
    gu_c, dn_c, w_c, ids = oracle_lib.compact_layer(gu, dn, w, retained)
    assert gu_c.shape == (8,) + gu.shape[1:] and w_c.shape == (8, w.shape[1])
    b = oracle_lib.moe_decode(xb, w_c, None, gu_c, dn_c, shape.top_k)
    assert np.array_equal(ids[b["idx"]], a["idx"])
    assert np.array_equal(b["gates"], a["gates"])
    assert np.array_equal(b["out"], a["out"])
    # with every logit tied (zero router) both forms must pick the lowest
    # original ids: the compact experts keep ascending original order
    z0 = np.zeros_like(w)
    a0 = oracle_lib.moe_decode(xb, z0, retained, gu, dn, shape.top_k)
    _, _, w0_c, ids0 = oracle_lib.compact_layer(gu, dn, z0, retained)
    b0 = oracle_lib.moe_decode(xb, w0_c, None, gu_c, dn_c, shape.top_k)
    assert np.array_equal(ids0[b0["idx"]], a0["idx"])
    assert np.array_equal(b0["out"], a0["out"])
    for bad in (np.array([1, 1, 2], np.int32), np.array([0, shape.num_experts], np.int32)):
        with pytest.raises(ValueError):
            oracle_lib.compact_layer(gu, dn, w, bad)


def test_full_pool_equals_unpruned(oracle_lib):
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=3)
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    a = oracle_lib.moe_decode(xb, w, None, gu, dn, shape.top_k)
    b = oracle_lib.moe_decode(xb, w, np.arange(shape.num_experts, dtype=np.int32)[::-1].copy(),
                              gu, dn, shape.top_k)
    for key in ("idx", "gates", "out"):
        assert np.array_equal(a[key], b[key])


# --------------------------------------------------------------------------
# top_k = 1 with a one-hot router reduces the layer to a dense SwiGLU FFN
# --------------------------------------------------------------------------
def _dense_swiglu(x64, gu64, d64):
    I = gu64.shape[0] // 2
    g = gu64[:I] @ x64
    u = gu64[I:] @ x64
    return d64 @ (g / (1.0 + np.exp(-g)) * u)


def test_top1_one_hot_router_is_dense_ffn(oracle_lib):
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=4)
    retained = synth.retained_set(shape.num_experts, 8, seed=2).numpy()
    e_star = int(retained[3])
    x, wr = synth.apply_popularity_bias(x, wr, torch.zeros(shape.num_experts))
    wr[e_star, -1] = 8.0
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    r = oracle_lib.moe_decode(xb, w, retained, gu, dn, 1)
    assert np.all(r["idx"][:, 0] == e_star)
    assert np.all(r["gates"] == 1.0)
    x64 = _bf16_to_f64(xb)
    ref = np.stack([_dense_swiglu(x64[t], _bf16_to_f64(gu[e_star]), _bf16_to_f64(dn[e_star]))
                    for t in range(x64.shape[0])])
    np.testing.assert_allclose(r["out"], ref, rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------
# Closed form: selection-matrix experts and exactly representable logits
# --------------------------------------------------------------------------
def test_closed_form_selection_experts_and_gates(oracle_lib):
    from tests.golden.closed_form import build_case, closed_form_out
    case = build_case()
    r = oracle_lib.moe_decode(case["x"], case["router_w"], case["retained"],
                              case["w_gate_up"], case["w_down"], case["k"])
    assert np.array_equal(r["idx"], case["expect_idx"])
    np.testing.assert_allclose(r["gates"], case["expect_gates"], rtol=1e-15, atol=0)
    np.testing.assert_allclose(r["out"], closed_form_out(case), rtol=1e-13, atol=1e-15)


def test_golden_fixture_reproduced(oracle_lib):
    import json
    import os
    from tests.golden.closed_form import build_case
    path = os.path.join(os.path.dirname(__file__), "golden", "closed_form_layer.json")
    with open(path) as f:
        gold = json.load(f)
    case = build_case()
    r = oracle_lib.moe_decode(case["x"], case["router_w"], case["retained"],
                              case["w_gate_up"], case["w_down"], case["k"])
    assert r["idx"].tolist() == gold["idx"]
    np.testing.assert_allclose(r["gates"], np.array(gold["gates"]), rtol=1e-15, atol=0)
    np.testing.assert_allclose(r["out"], np.array(gold["out"]), rtol=1e-14, atol=1e-16)


# --------------------------------------------------------------------------
# Token subsets: the layer is a per-token gate-weighted sum (Sec. 3.1), so the
# layer evaluated for a subset of the batch gives exactly those tokens' rows
# --------------------------------------------------------------------------
def test_token_subset_rows_equal_whole_batch_rows(oracle_lib):
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=9)
    retained = synth.retained_set(shape.num_experts, 8, seed=2).numpy()
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    k = shape.top_k
    whole = oracle_lib.moe_decode(xb, w, retained, gu, dn, k)
    T = np.array([7, 2, 5, 0, 8], np.int32)          # unsorted, not contiguous
    part = oracle_lib.moe_decode_sampled(xb, w, retained, gu, dn, k, T)
    assert np.array_equal(part["idx"], whole["idx"])
    assert np.array_equal(part["out"], whole["out"][T])
    # each sampled row against a float64 numpy evaluation of its own token
    x64 = _bf16_to_f64(xb)
    for r, t in enumerate(T):
        ref = sum(part["gates"][t, j] * _dense_swiglu(x64[t], _bf16_to_f64(gu[e]), _bf16_to_f64(dn[e]))
                  for j, e in enumerate(part["idx"][t]))
        np.testing.assert_allclose(part["out"][r], ref, rtol=1e-10, atol=1e-13)
    # with the shared expert (Sec. 3.3) each row also carries its own token's
    # gate and shared term
    se_gu, se_dn, w_sg = _shared_expert(5, 64)
    whole_s = oracle_lib.moe_decode_shared(xb, w, retained, gu, dn, k, w_sg, se_gu, se_dn)
    part_s = oracle_lib.moe_decode_shared(xb, w, retained, gu, dn, k, w_sg, se_gu, se_dn, tokens=T)
    assert np.array_equal(part_s["shared_gate"], whole_s["shared_gate"][T])
    assert np.array_equal(part_s["out"], whole_s["out"][T])
    s_ref = 1.0 / (1.0 + np.exp(-(x64[T] @ w_sg.astype(np.float64))))
    np.testing.assert_allclose(part_s["shared_gate"], s_ref, rtol=1e-5)


# --------------------------------------------------------------------------
# Batch-permutation invariance
# --------------------------------------------------------------------------
def test_batch_permutation_invariance(oracle_lib):
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=6)
    retained = synth.retained_set(shape.num_experts, 8, seed=2).numpy()
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    a = oracle_lib.moe_decode(xb, w, retained, gu, dn, shape.top_k)
    p = np.random.default_rng(5).permutation(xb.shape[0])
    b = oracle_lib.moe_decode(np.ascontiguousarray(xb[p]), w, retained, gu, dn, shape.top_k)
    for key in ("idx", "gates", "out"):
        assert np.array_equal(a[key][p], b[key])
    ga = oracle_lib.group_by_expert(a["idx"], shape.num_experts)
    gb = oracle_lib.group_by_expert(b["idx"], shape.num_experts)
    assert np.array_equal(ga["counts"], gb["counts"])
    assert np.array_equal(ga["union_ids"], gb["union_ids"])
    # grouped slots carry the same expert sequence; tokens map through p
    k = shape.top_k
    ea = a["idx"].reshape(-1)[ga["perm"]]
    eb = b["idx"].reshape(-1)[gb["perm"]]
    assert np.array_equal(ea, eb)


# --------------------------------------------------------------------------
# Grouping by expert: structure, stable sort, union by enumeration, Eq. 1
# --------------------------------------------------------------------------
def _random_subsets(rng, B, k, pool):
    return np.stack([rng.choice(pool, size=k, replace=False) for _ in range(B)]).astype(np.int32)


@pytest.mark.parametrize("B,k,E", [(1, 1, 4), (5, 2, 16), (33, 8, 128), (64, 8, 128), (3, 4, 4)])
def test_grouping_structure_and_stable_sort(oracle_lib, B, k, E):
    rng = np.random.default_rng(B * 131 + k)
    idx = _random_subsets(rng, B, k, np.arange(E))
    g = oracle_lib.group_by_expert(idx, E)
    flat = idx.reshape(-1)
    assert g["counts"].sum() == B * k
    assert g["offsets"][0] == 0 and g["offsets"][-1] == B * k
    assert np.all(np.diff(g["offsets"]) == g["counts"])
    assert np.array_equal(np.sort(g["perm"]), np.arange(B * k))
    assert np.array_equal(g["pos"][g["perm"]], np.arange(B * k))
    # a stable sort of the flat slots by expert id is the grouped order
    assert np.array_equal(g["perm"], np.argsort(flat, kind="stable"))
    # union by set enumeration
    assert g["union_ids"].tolist() == sorted(set(flat.tolist()))
    assert g["union_size"] == len(set(flat.tolist()))
    for e in range(E):
        seg = g["perm"][g["offsets"][e]:g["offsets"][e + 1]]
        assert np.all(flat[seg] == e)
        assert np.all(np.diff(seg // k) > 0)     # token ascending within an expert


@pytest.mark.parametrize("m_prime,B", [(128, 8), (64, 16), (32, 4), (96, 1)])
def test_union_size_matches_eq1_expectation(oracle_lib, m_prime, B):
    # Eq. 1: with each token drawing k distinct experts uniformly and
    # independently, E[distinct] = m'[1 - (1 - k/m')^B] exactly.
    k, E, draws = 8, 128, 2000
    rng = np.random.default_rng(m_prime * 7 + B)
    pool = np.sort(rng.choice(E, size=m_prime, replace=False))
    u = np.array([oracle_lib.group_by_expert(_random_subsets(rng, B, k, pool), E)["union_size"]
                  for _ in range(draws)], np.float64)
    expect = m_prime * (1.0 - (1.0 - k / m_prime) ** B)
    sem = max(u.std(ddof=1), 1e-9) / math.sqrt(draws)
    assert abs(u.mean() - expect) <= 4 * sem + 1e-9, (u.mean(), expect, sem)


# --------------------------------------------------------------------------
# Shared expert (Sec. 3.3): always-on SwiGLU expert under a sigmoid gate
# --------------------------------------------------------------------------
def _shared_expert(seed, I_s, H=256):
    one = synth.LayerShape(hidden=H, num_experts=1, inter=I_s, top_k=1)
    gu, dn = synth.expert_weights(one, seed)
    g = torch.Generator().manual_seed(seed + 17)
    w_sg = (torch.randn(H, generator=g) * 0.05).to(torch.float32)
    return _bits(gu[0]), _bits(dn[0]), w_sg.numpy()


def _shared_only(oracle_lib, xb, w_sg, gu, dn):
    out = np.zeros((xb.shape[0], xb.shape[1]), np.float64)
    s = oracle_lib.shared_expert_add(xb, w_sg, gu, dn, out)
    return out, s


def test_shared_expert_gate_is_sigmoid_of_canonical_logit(oracle_lib):
    x, _, _, _ = _tiny_layer(B=5)
    xb = _bits(x)
    gu, dn, w_sg = _shared_expert(3, 64)
    _, s = _shared_only(oracle_lib, xb, w_sg, gu, dn)
    x64 = _bf16_to_f64(xb)
    z_exact = x64 @ w_sg.astype(np.float64)
    absdot = np.abs(x64) @ np.abs(w_sg.astype(np.float64))
    n_ops = xb.shape[1] // 32 + 5
    gamma = n_ops * 2.0 ** -24 / (1 - n_ops * 2.0 ** -24)
    # |ds/dz| <= 1/4: the gate is the sigmoid of z within the fp32 sum's error
    ref = 1.0 / (1.0 + np.exp(-z_exact))
    assert np.all(np.abs(s - ref) <= 0.25 * gamma * absdot + 1e-15)
    assert np.all((s > 0) & (s < 1))


def test_shared_expert_saturated_gates(oracle_lib):
    # gate logit -1000: the shared term vanishes exactly; +1000: the whole
    # expert is added, equal to a dense numpy SwiGLU
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=4)
    x, wr = synth.apply_popularity_bias(x, wr, torch.zeros(shape.num_experts))
    xb, w, gu_r, dn_r = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    retained = synth.retained_set(shape.num_experts, 8, seed=2).numpy()
    gu, dn, w_sg = _shared_expert(5, 64)
    w_sg = np.zeros_like(w_sg)
    routed = oracle_lib.moe_decode(xb, w, retained, gu_r, dn_r, 2)["out"]
    w_sg[-1] = -1000.0
    off = oracle_lib.moe_decode_shared(xb, w, retained, gu_r, dn_r, 2, w_sg, gu, dn)
    assert np.all(off["shared_gate"] == 0.0)
    assert np.array_equal(off["out"], routed)
    w_sg[-1] = 1000.0
    on = oracle_lib.moe_decode_shared(xb, w, retained, gu_r, dn_r, 2, w_sg, gu, dn)
    assert np.all(on["shared_gate"] == 1.0)
    x64 = _bf16_to_f64(xb)
    dense = np.stack([_dense_swiglu(x64[t], _bf16_to_f64(gu), _bf16_to_f64(dn)) for t in range(4)])
    np.testing.assert_allclose(on["out"] - routed, dense, rtol=1e-9, atol=1e-12)


def test_shared_expert_twice_width_is_sum_of_halves(oracle_lib):
    # Sec. 3.3: two shared experts under one gate are one expert of twice the
    # intermediate width ([gate1; gate2; up1; up2] rows, [down1 | down2] columns)
    x, _, _, _ = _tiny_layer(B=3)
    xb = _bits(x)
    gu1, dn1, w_sg = _shared_expert(7, 32)
    gu2, dn2, _ = _shared_expert(8, 32)
    I = 32
    gu = np.concatenate([gu1[:I], gu2[:I], gu1[I:], gu2[I:]], axis=0)
    dn = np.concatenate([dn1, dn2], axis=1)
    both, s = _shared_only(oracle_lib, xb, w_sg, gu, dn)
    a, _ = _shared_only(oracle_lib, xb, w_sg, gu1, dn1)
    b, _ = _shared_only(oracle_lib, xb, w_sg, gu2, dn2)
    np.testing.assert_allclose(both, a + b, rtol=1e-12, atol=1e-15)
    # the second expert starts with a zero down projection: the layer output
    # is unchanged at initialisation
    dn_init = np.concatenate([dn1, np.zeros_like(dn2)], axis=1)
    init, _ = _shared_only(oracle_lib, xb, w_sg, gu, dn_init)
    assert np.array_equal(init, a)


# --------------------------------------------------------------------------
# Expert-importance statistics and the retained set (Sec. 2.3, Sec. 3.1)
# --------------------------------------------------------------------------
def test_expert_stats_totals_and_one_hot_router(oracle_lib):
    # every token makes k selections whose gates sum to one
    shape = synth.TINY
    x, wr, w_gu, w_d = _tiny_layer(B=12)
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    st = oracle_lib.expert_stats(xb, w, gu, dn, 2)
    assert st[:, 0].sum() == 12 * 2
    assert abs(st[:, 1].sum() - 12.0) < 1e-12
    assert np.all(st >= 0) and np.all(st[st[:, 0] == 0] == 0)
    # statistics accumulate over calibration batches
    st2 = oracle_lib.expert_stats(xb, w, gu, dn, 2, stats=st.copy())
    np.testing.assert_allclose(st2, 2 * st, rtol=1e-15, atol=0)
    # top-1 one-hot router: every token goes to e* with gate 1, so EAN is the
    # sum of the dense SwiGLU output norms and REAP is EAN / count
    e_star = 5
    x1, wr1 = synth.apply_popularity_bias(x, wr, torch.zeros(shape.num_experts))
    wr1[e_star, -1] = 8.0
    xb1, w1 = _bits(x1), wr1.numpy()
    st1 = oracle_lib.expert_stats(xb1, w1, gu, dn, 1)
    x64 = _bf16_to_f64(xb1)
    norms = [np.linalg.norm(_dense_swiglu(x64[t], _bf16_to_f64(gu[e_star]), _bf16_to_f64(dn[e_star])))
             for t in range(12)]
    assert st1[e_star, 0] == 12 and st1[e_star, 1] == 12.0
    np.testing.assert_allclose(st1[e_star, 2], sum(norms), rtol=1e-11)
    np.testing.assert_allclose(st1[e_star, 3], sum(norms), rtol=1e-11)
    assert np.all(np.delete(st1, e_star, axis=0) == 0)
    ids = oracle_lib.select_retained(st1, 1, "reap")
    assert list(ids) == [e_star]
    # zero router: every token selects experts 0..k-1 with gate exactly 1/k,
    # so each REAP numerator is its EAN / k and each mass is count / k
    k = 4
    st0 = oracle_lib.expert_stats(xb, np.zeros_like(w), gu, dn, k)
    assert np.all(st0[:k, 0] == 12) and np.all(st0[k:] == 0)
    np.testing.assert_allclose(st0[:k, 1], 12 / k, rtol=1e-14)
    np.testing.assert_allclose(st0[:k, 3], st0[:k, 2] / k, rtol=1e-13)


def test_routing_mass_takes_gates_of_selected_experts_only(oracle_lib):
    # Sec. 2.3 says routing mass aggregates gate probabilities.  The reading
    # here sums each token's renormalised gates over its k selections, the
    # weights the layer actually applies (the same gates REAP multiplies the
    # output norms by).  Summing the pool softmax over every token instead
    # would credit experts that are never selected: here expert 9 is every
    # token's runner-up at top-1, with a pool probability near one half and
    # a routing mass of exactly zero, so the two readings keep different sets.
    shape = synth.TINY
    E, B = shape.num_experts, 10
    x, _, w_gu, w_d = _tiny_layer(B=B)
    bias = torch.full((E,), -5.0)
    bias[0], bias[9] = 1.0, 0.99
    x, wr = synth.apply_popularity_bias(x, torch.zeros((E, shape.hidden)), bias)
    xb, w, gu, dn = _bits(x), wr.numpy(), _bits(w_gu), _bits(w_d)
    st = oracle_lib.expert_stats(xb, w, gu, dn, 1)
    assert st[0, 0] == B and st[0, 1] == B
    assert np.all(st[1:] == 0)
    z = oracle_lib.router_logits(xb, w).astype(np.float64)
    p = np.exp(z - z.max(1, keepdims=True))
    p /= p.sum(1, keepdims=True)
    pool_mass = p.sum(0)
    assert pool_mass[9] > 0.45 * B
    assert list(oracle_lib.select_retained(st, 2, "mass")) == [0, 1]        # ties to the lowest id
    assert sorted(np.argsort(-pool_mass, kind="stable")[:2].tolist()) == [0, 9]


@pytest.mark.parametrize("seed", [0, 1])
def test_select_retained_matches_brute_force_with_ties(oracle_lib, seed):
    rng = np.random.default_rng(seed)
    E = 24
    st = np.zeros((E, 4))
    st[:, 0] = rng.integers(0, 4, E)
    # few distinct values: many ties
    st[:, 1] = rng.integers(0, 3, E) * 0.5
    st[:, 2] = rng.integers(0, 3, E) * 0.25
    st[:, 3] = st[:, 2] * st[:, 1]
    for crit in ("mass", "ean", "reap"):
        if crit == "mass":
            score = st[:, 1]
        elif crit == "ean":
            score = st[:, 2]
        else:
            score = np.where(st[:, 0] > 0, st[:, 3] / np.maximum(st[:, 0], 1), 0.0)
        for m in (0, 1, 7, E):
            # brute force: sort by (score desc, id asc), keep m, report ascending
            order = sorted(range(E), key=lambda e: (-score[e], e))[:m]
            assert list(oracle_lib.select_retained(st, m, crit)) == sorted(order)
