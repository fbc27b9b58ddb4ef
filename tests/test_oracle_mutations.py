"""Planted mistakes in the oracle must each fail at least one pin.

Every mutation edits a copy of the oracle's C source on the CPU (a dropped
term, a swapped operand, a wrong sign, index or tie-break), builds it, swaps it
in and runs the pin functions of test_oracle_pins; at least one must fail.
"""
import numpy as np
import pytest

import oracle
from tests import test_oracle_pins as pins

MUTATIONS = {
    # router logits: drop the last element of each 4-wide group
    "logit_drop_term": ("for (int q = 0; q < 4; ++q) {", "for (int q = 0; q < 3; ++q) {"),
    # router logits: read the router row of the wrong expert
    "logit_wrong_row": ("wr[(size_t)e * H + h], p[l]);", "wr[(size_t)((e + 1) % E) * H + h], p[l]);"),
    # Eq. 2 ignored: masked experts keep their logit
    "mask_ignored": ("zm[e] = in_set[e] ? z[(size_t)t * E + e] : -INFINITY;", "zm[e] = z[(size_t)t * E + e];"),
    # tie-break to the highest id
    "tie_highest_id": ("if (best < 0 || zm[e] > zm[best]) best = e;", "if (best < 0 || zm[e] >= zm[best]) best = e;"),
    # gates: softmax with the wrong sign
    "gate_sign": ("exp((double)zm[idx[(size_t)t * k + j]] - z1) / denom;", "exp(z1 - (double)zm[idx[(size_t)t * k + j]]) / denom;"),
    # SwiGLU: gate and up swapped
    "swap_gate_up": ("a[i] = g / (1.0 + exp(-g)) * u;", "a[i] = u / (1.0 + exp(-u)) * g;"),
    # SiLU sign error
    "silu_sign": ("a[i] = g / (1.0 + exp(-g)) * u;", "a[i] = g / (1.0 + exp(g)) * u;"),
    # down projection transposed (in x out instead of out x in)
    "down_transposed": ("acc += (double)bf16_to_float(wd[(size_t)h * I + i]) * a[i];",
                        "acc += (double)bf16_to_float(wd[(size_t)i * H + h]) * a[i];"),
    # combine: gates not applied
    "combine_no_gate": ("for (int h = 0; h < H; ++h) o[h] += g * y[h];", "for (int h = 0; h < H; ++h) o[h] += y[h];"),
    # shared expert: sigmoid with the wrong sign
    "shared_gate_sign": ("double s = 1.0 / (1.0 + exp(-(double)z));", "double s = 1.0 / (1.0 + exp((double)z));"),
    # shared expert: gate not applied
    "shared_gate_dropped": ("for (int h = 0; h < H; ++h) o[h] += s * y[h];", "for (int h = 0; h < H; ++h) o[h] += y[h];"),
    # statistics: activation norm squared instead of the norm
    "stats_norm_squared": ("stats[(size_t)e * 4 + 2] += nrm;", "stats[(size_t)e * 4 + 2] += n2;"),
    # statistics: REAP without the gate
    "stats_reap_no_gate": ("stats[(size_t)e * 4 + 3] += g * nrm;", "stats[(size_t)e * 4 + 3] += nrm;"),
    # selection: ties to the highest id
    "select_tie_highest": ("if (!taken[e] && (best < 0 || score[e] > score[best])) best = e;",
                           "if (!taken[e] && (best < 0 || score[e] >= score[best])) best = e;"),
    # grouping: offsets off by one expert
    "offsets_shift": ("offsets[e + 1] = offsets[e] + counts[e];", "offsets[e + 1] = offsets[e] + counts[e > 0 ? e - 1 : 0];"),
    # combine for a token subset: row r computed for token r instead of tokens[r]
    "combine_token_index": ("    int t = tokens[r];\n    double *o = out + (size_t)r * H;",
                            "    int t = r;\n    double *o = out + (size_t)r * H;"),
    # shared expert for a token subset: the same slip
    "shared_token_index": ("    int t = tokens[r];\n    float z;", "    int t = r;\n    float z;"),
    # grouping: token order reversed inside an expert
    "perm_token_desc": ("for (int t = 0; t < B; ++t)\n    for (int j = 0; j < k; ++j) {\n      int s = t * k + j;",
                        "for (int t = B - 1; t >= 0; --t)\n    for (int j = 0; j < k; ++j) {\n      int s = t * k + j;"),
}

PIN_FUNCS = [
    (pins.test_logits_within_summation_error_bound, ()),
    (pins.test_logits_exact_on_representable_inputs, ()),
    (pins.test_topk_matches_brute_force_with_ties, (0,)),
    (pins.test_topk_matches_brute_force_with_ties, (3,)),
    (pins.test_zero_router_selects_lowest_retained_ids_with_equal_gates, ()),
    (pins.test_gates_equal_pool_softmax_renormalised_over_topk, ()),
    (pins.test_top1_one_hot_router_is_dense_ffn, ()),
    (pins.test_closed_form_selection_experts_and_gates, ()),
    (pins.test_grouping_structure_and_stable_sort, (33, 8, 128)),
    (pins.test_shared_expert_gate_is_sigmoid_of_canonical_logit, ()),
    (pins.test_shared_expert_saturated_gates, ()),
    (pins.test_shared_expert_twice_width_is_sum_of_halves, ()),
    (pins.test_expert_stats_totals_and_one_hot_router, ()),
    (pins.test_select_retained_matches_brute_force_with_ties, (0,)),
    (pins.test_token_subset_rows_equal_whole_batch_rows, ()),
]


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name):
    old, new = MUTATIONS[name]
    src = oracle.source_text()
    assert src.count(old) == 1, f"mutation anchor for {name} not found exactly once"
    path = oracle.build_variant(src.replace(old, new), name)
    failures = 0
    with oracle.swapped_library(path):
        for fn, args in PIN_FUNCS:
            try:
                fn(oracle, *args)
            except (AssertionError, ValueError, IndexError):
                failures += 1
    assert failures > 0, f"no pin caught mutation {name}"


# The pruned-checkpoint compaction is numpy in oracle/__init__.py: its planted
# mistakes replace the Python function.
def _compact_unsorted(w_gate_up, w_down, router_w, retained):
    # the retained experts kept in the caller's order, not ascending id
    ids = np.asarray(retained, np.int64).ravel()
    return w_gate_up[ids], w_down[ids], router_w[ids], ids.astype(np.int32)


def _compact_down_rows_shifted(w_gate_up, w_down, router_w, retained):
    # the down projection taken from the neighbouring retained expert
    ids = np.sort(np.asarray(retained, np.int64).ravel())
    return w_gate_up[ids], w_down[np.roll(ids, 1)], router_w[ids], ids.astype(np.int32)


def _compact_router_rows_of_pool_order(w_gate_up, w_down, router_w, retained):
    # the first m' router rows instead of the retained experts' rows
    ids = np.sort(np.asarray(retained, np.int64).ravel())
    return w_gate_up[ids], w_down[ids], router_w[:ids.size], ids.astype(np.int32)


PY_MUTATIONS = {
    "compact_unsorted": _compact_unsorted,
    "compact_down_rows_shifted": _compact_down_rows_shifted,
    "compact_router_rows_of_pool_order": _compact_router_rows_of_pool_order,
}


@pytest.mark.parametrize("name", sorted(PY_MUTATIONS))
def test_planted_compaction_mistake_is_caught(name, monkeypatch):
    monkeypatch.setattr(oracle, "compact_layer", PY_MUTATIONS[name])
    with pytest.raises((AssertionError, ValueError, IndexError)):
        pins.test_masked_router_equals_pruned_checkpoint(oracle)
