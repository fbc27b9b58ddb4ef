"""The OpenMP build of the oracle (used only to time it on all host cores)
computes exactly what the plain build computes: it splits the tokens of the
expert/combine step across threads and leaves each token's arithmetic and its
order alone, so every selection, gate and output must be bit-identical."""
import os

import numpy as np
import pytest

import oracle
from paper_2609_34117_gb300 import synth


def test_openmp_build_is_bit_identical_to_the_plain_build(monkeypatch):
    monkeypatch.setenv("OMP_NUM_THREADS", "4")
    try:
        path = oracle.build_openmp()
    except Exception as exc:   # no OpenMP in this toolchain: nothing to compare
        pytest.skip(f"no OpenMP build: {exc}")
    shape = synth.TINY
    w_gu, w_d = synth.expert_weights(shape, 5)
    wr = synth.router_weight(shape, 5).numpy()
    x = synth.bf16_bits(synth.hidden_states(37, shape, 6))
    gu, dn = synth.bf16_bits(w_gu), synth.bf16_bits(w_d)
    retained = synth.retained_set(shape.num_experts, 8, 7, shuffle=True).numpy()
    tokens = np.array([36, 0, 17, 5, 22], dtype=np.int32)
    plain = oracle.moe_decode(x, wr, retained, gu, dn, shape.top_k)
    plain_s = oracle.moe_decode_sampled(x, wr, retained, gu, dn, shape.top_k, tokens)
    with oracle.swapped_library(path):
        threads = oracle.num_threads()
        omp = oracle.moe_decode(x, wr, retained, gu, dn, shape.top_k)
        omp_s = oracle.moe_decode_sampled(x, wr, retained, gu, dn, shape.top_k, tokens)
    if (os.cpu_count() or 1) > 1:
        assert threads > 1
    for key in ("idx", "gates", "out"):
        assert np.array_equal(plain[key], omp[key]), key
        assert np.array_equal(plain_s[key], omp_s[key]), key
