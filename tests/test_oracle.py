"""Pins for the fp64 oracle (CPU only).

Each test checks the oracle against something other than itself: closed
forms, a hand-derived worked example, an independent dense formulation through
scipy.special on tiny inputs, or invariants that the definition fixes
(chunk consistency, head grouping, sequence permutation, empty rows).
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from helpers import bf16_bits_to_f64, dense_reference, f32_to_bf16_bits, random_bf16

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "worked_example.json")


def _run(q, k, v, cu_q, cu_k, Hq, Hkv, scale):
    d = q.shape[-1]
    return oracle.attention(q, k, v, cu_q, cu_k, Hq, Hkv, d, scale, n_threads=2)


def _closed(expr):
    return float(eval(expr, {"__builtins__": {}}, {"e": math.e, "log": math.log, "inf": math.inf}))


@pytest.mark.parametrize("case", range(3))
def test_worked_example(case):
    spec = json.load(open(GOLDEN))["cases"][case]
    q = f32_to_bf16_bits(np.array(spec["q"], dtype=np.float32))
    k = f32_to_bf16_bits(np.array(spec["k"], dtype=np.float32))
    v = f32_to_bf16_bits(np.array(spec["v"], dtype=np.float32))
    # the example values are exact in bf16
    np.testing.assert_array_equal(bf16_bits_to_f64(q), np.array(spec["q"]))
    o, lse = _run(q, k, v, spec["cu_q"], spec["cu_k"], spec["Hq"], spec["Hkv"], spec["scale"])
    for e in spec["expected"]:
        want_o = [_closed(x) for x in e["o"]]
        want_lse = _closed(e["lse"])
        np.testing.assert_allclose(o[e["token"], e["head"]], want_o, rtol=0, atol=1e-14)
        if math.isinf(want_lse):
            assert lse[e["token"], e["head"]] == want_lse
        else:
            assert abs(lse[e["token"], e["head"]] - want_lse) < 1e-14


def test_length_one_row_is_its_value_row():
    rng = np.random.default_rng(1)
    Hq, Hkv, d = 4, 2, 64
    lens = [1, 1, 1]
    cu = np.concatenate([[0], np.cumsum(lens)])
    q, k, v = (random_bf16(rng, (3, Hq, d)), random_bf16(rng, (3, Hkv, d)),
               random_bf16(rng, (3, Hkv, d)))
    scale = 0.125
    o, lse = _run(q, k, v, cu, cu, Hq, Hkv, scale)
    qf, kf, vf = bf16_bits_to_f64(q), bf16_bits_to_f64(k), bf16_bits_to_f64(v)
    for t in range(3):
        for h in range(Hq):
            g = h // (Hq // Hkv)
            np.testing.assert_array_equal(o[t, h], vf[t, g])
            want = scale * math.fsum(qf[t, h] * kf[t, g])
            assert abs(lse[t, h] - want) <= 1e-13 * max(1.0, abs(want))


def test_constant_values_give_that_constant():
    rng = np.random.default_rng(2)
    Hq, Hkv, d = 4, 1, 16
    lens = [5, 33, 2]
    cu = np.concatenate([[0], np.cumsum(lens)])
    T = cu[-1]
    q, k = random_bf16(rng, (T, Hq, d), 2.0), random_bf16(rng, (T, Hkv, d), 2.0)
    v = f32_to_bf16_bits(np.full((T, Hkv, d), 0.75, dtype=np.float32))
    o, _ = _run(q, k, v, cu, cu, Hq, Hkv, 0.25)
    np.testing.assert_allclose(o, 0.75, rtol=0, atol=1e-14)


def test_zero_queries_average_visible_values():
    rng = np.random.default_rng(3)
    Hq, Hkv, d = 2, 2, 8
    lq, lk = [6, 3], [9, 3]  # first sequence is a chunk with a 3-token prefix
    cu_q, cu_k = np.concatenate([[0], np.cumsum(lq)]), np.concatenate([[0], np.cumsum(lk)])
    q = np.zeros((cu_q[-1], Hq, d), dtype=np.uint16)  # +0.0 in bf16
    k, v = random_bf16(rng, (cu_k[-1], Hkv, d)), random_bf16(rng, (cu_k[-1], Hkv, d))
    o, lse = _run(q, k, v, cu_q, cu_k, Hq, Hkv, 0.3)
    vf = bf16_bits_to_f64(v)
    for s in range(2):
        delta = lk[s] - lq[s]
        for i in range(lq[s]):
            n_vis = min(i + delta + 1, lk[s])
            for h in range(Hq):
                rows = vf[cu_k[s]:cu_k[s] + n_vis, h]
                want = np.array([math.fsum(rows[:, c]) / n_vis for c in range(d)])
                np.testing.assert_allclose(o[cu_q[s] + i, h], want, rtol=0, atol=1e-14)
                assert abs(lse[cu_q[s] + i, h] - math.log(n_vis)) < 1e-14


SHAPES = [
    # (q_lens, k_lens, Hq, Hkv, d)
    ([1, 17, 64], [1, 17, 64], 4, 2, 64),
    ([5, 0, 9], [12, 0, 9], 6, 3, 16),          # chunk + empty sequence
    ([7, 4], [3, 4], 4, 4, 8),                   # more queries than keys in sequence 0
    ([33], [70], 8, 1, 32),                      # multi-query, long prefix
]


@pytest.mark.parametrize("shape", SHAPES)
def test_matches_dense_scipy_formulation(shape):
    lq, lk, Hq, Hkv, d = shape
    rng = np.random.default_rng(sum(lq) + 7 * Hq)
    cu_q, cu_k = np.concatenate([[0], np.cumsum(lq)]), np.concatenate([[0], np.cumsum(lk)])
    q = random_bf16(rng, (cu_q[-1], Hq, d), 1.5)
    k = random_bf16(rng, (cu_k[-1], Hkv, d), 1.5)
    v = random_bf16(rng, (cu_k[-1], Hkv, d))
    scale = 1.0 / math.sqrt(d)
    o, lse = _run(q, k, v, cu_q, cu_k, Hq, Hkv, scale)
    o_ref, lse_ref = dense_reference(q, k, v, cu_q, cu_k, Hq, Hkv, scale)
    np.testing.assert_allclose(o, o_ref, rtol=0, atol=1e-12)
    fin = np.isfinite(lse_ref)
    np.testing.assert_array_equal(np.isfinite(lse), fin)
    np.testing.assert_allclose(lse[fin], lse_ref[fin], rtol=0, atol=1e-12)
    assert np.all(lse[~fin] == -np.inf)


def test_chunk_consistency_pins_bottom_right_alignment():
    """The last m rows of a full causal prompt equal a chunk of m queries over all keys."""
    rng = np.random.default_rng(5)
    Hq, Hkv, d, n, m = 4, 2, 32, 40, 11
    q = random_bf16(rng, (n, Hq, d))
    k, v = random_bf16(rng, (n, Hkv, d)), random_bf16(rng, (n, Hkv, d))
    o_full, lse_full = _run(q, k, v, [0, n], [0, n], Hq, Hkv, 0.2)
    o_chunk, lse_chunk = _run(q[n - m:], k, v, [0, m], [0, n], Hq, Hkv, 0.2)
    np.testing.assert_array_equal(o_chunk, o_full[n - m:])
    np.testing.assert_array_equal(lse_chunk, lse_full[n - m:])


def test_head_groups_are_contiguous():
    """GQA equals multi-head attention with each kv head repeated for its G query heads."""
    rng = np.random.default_rng(6)
    Hq, Hkv, d, n = 4, 2, 16, 12
    q = random_bf16(rng, (n, Hq, d))
    k, v = random_bf16(rng, (n, Hkv, d)), random_bf16(rng, (n, Hkv, d))
    o_gqa, lse_gqa = _run(q, k, v, [0, n], [0, n], Hq, Hkv, 0.25)
    rep = [0, 0, 1, 1]
    o_mha, lse_mha = _run(q, k[:, rep], v[:, rep], [0, n], [0, n], Hq, Hq, 0.25)
    np.testing.assert_array_equal(o_gqa, o_mha)
    np.testing.assert_array_equal(lse_gqa, lse_mha)
    # the interleaved reading (h -> h mod Hkv) gives different numbers
    o_int, _ = _run(q, k[:, [0, 1, 0, 1]], v[:, [0, 1, 0, 1]], [0, n], [0, n], Hq, Hq, 0.25)
    assert np.abs(o_int - o_gqa).max() > 1e-3


def test_sequence_permutation_permutes_rows():
    rng = np.random.default_rng(8)
    Hq, Hkv, d = 2, 1, 16
    lq, lk = [3, 8, 5], [6, 8, 5]
    cu_q, cu_k = np.concatenate([[0], np.cumsum(lq)]), np.concatenate([[0], np.cumsum(lk)])
    q = random_bf16(rng, (cu_q[-1], Hq, d))
    k, v = random_bf16(rng, (cu_k[-1], Hkv, d)), random_bf16(rng, (cu_k[-1], Hkv, d))
    o, lse = _run(q, k, v, cu_q, cu_k, Hq, Hkv, 0.25)
    perm = [2, 0, 1]
    qp = np.concatenate([q[cu_q[s]:cu_q[s + 1]] for s in perm])
    kp = np.concatenate([k[cu_k[s]:cu_k[s + 1]] for s in perm])
    vp = np.concatenate([v[cu_k[s]:cu_k[s + 1]] for s in perm])
    cu_qp = np.concatenate([[0], np.cumsum([lq[s] for s in perm])])
    cu_kp = np.concatenate([[0], np.cumsum([lk[s] for s in perm])])
    op, lsep = _run(qp, kp, vp, cu_qp, cu_kp, Hq, Hkv, 0.25)
    np.testing.assert_array_equal(op, np.concatenate([o[cu_q[s]:cu_q[s + 1]] for s in perm]))
    np.testing.assert_array_equal(lsep, np.concatenate([lse[cu_q[s]:cu_q[s + 1]] for s in perm]))


def test_rows_without_keys_are_zero_with_minus_infinity_lse():
    rng = np.random.default_rng(9)
    Hq, Hkv, d = 2, 2, 8
    q = random_bf16(rng, (5, Hq, d))
    k, v = random_bf16(rng, (2, Hkv, d)), random_bf16(rng, (2, Hkv, d))
    o, lse = _run(q, k, v, [0, 5], [0, 2], Hq, Hkv, 1.0)
    # delta = -3: rows 0..2 see nothing, row 3 sees key 0, row 4 sees keys 0..1
    assert np.all(o[:3] == 0) and np.all(lse[:3] == -np.inf)
    assert np.all(np.isfinite(lse[3:]))


def test_selected_rows_match_full_run():
    rng = np.random.default_rng(10)
    Hq, Hkv, d = 4, 2, 32
    lq = [9, 30, 1]
    cu = np.concatenate([[0], np.cumsum(lq)])
    q = random_bf16(rng, (cu[-1], Hq, d))
    k, v = random_bf16(rng, (cu[-1], Hkv, d)), random_bf16(rng, (cu[-1], Hkv, d))
    o, lse = _run(q, k, v, cu, cu, Hq, Hkv, 0.2)
    tok = np.array([0, 8, 9, 38, 39, 20])
    hd = np.array([3, 0, 1, 2, 3, 1])
    o_r, lse_r = oracle.attention_rows(q, k, v, cu, cu, Hq, Hkv, d, 0.2, tok, hd, n_threads=3)
    np.testing.assert_array_equal(o_r, o[tok, hd])
    np.testing.assert_array_equal(lse_r, lse[tok, hd])
