"""Pins of the QCTS oracle (section "Question Contrastive Teacher Selection", Eq. 1-2)
against library routines, closed forms, hand-worked cases and invariants."""
import math

import numpy as np
import pytest
from scipy.spatial.distance import jensenshannon
from scipy.stats import entropy

from oracle import qcts_oracle as Q
from paper_2608_06411_gb300 import workloads as W


def _dirichlet(rng, n, zeros=0):
    p = rng.gamma(0.5, size=n)
    if zeros:
        p[rng.choice(n, zeros, replace=False)] = 0.0
    return p / p.sum()


def test_js_matches_scipy_and_entropy_identity():
    rng = np.random.default_rng(1)
    for n, z in [(2, 0), (7, 2), (576, 40), (2880, 0)]:
        p, q = _dirichlet(rng, n, z), _dirichlet(rng, n, z)
        js = Q.js_divergence(p, q)
        # scipy returns the square root of the divergence (natural log by default)
        assert js == pytest.approx(jensenshannon(p, q) ** 2, rel=1e-10, abs=1e-15)
        m = 0.5 * (p + q)
        assert js == pytest.approx(entropy(m) - 0.5 * (entropy(p) + entropy(q)), rel=1e-9, abs=1e-15)


def test_js_closed_forms():
    p = np.array([1.0, 0.0])
    q = np.array([0.5, 0.5])
    # m = (3/4, 1/4): KL(p||m) = ln(4/3), KL(q||m) = ln(4/3)/2, JS = 3/4 ln(4/3)
    assert Q.js_divergence(p, q) == pytest.approx(0.75 * math.log(4.0 / 3.0), rel=1e-14)
    assert Q.js_divergence(q, p) == pytest.approx(0.75 * math.log(4.0 / 3.0), rel=1e-14)
    # disjoint supports: ln 2 (the maximum); identical: 0
    assert Q.js_divergence(np.array([0.3, 0.7, 0, 0]), np.array([0, 0, 0.9, 0.1])) == pytest.approx(math.log(2.0))
    r = np.array([0.1, 0.2, 0.7])
    assert Q.js_divergence(r, r) == 0.0
    rng = np.random.default_rng(2)
    for _ in range(50):
        a, b = _dirichlet(rng, 9, 3), _dirichlet(rng, 9, 3)
        v = Q.js_divergence(a, b)
        assert 0.0 <= v <= math.log(2.0) + 1e-15
        assert v == pytest.approx(Q.js_divergence(b, a), rel=1e-13)


def test_eq1_hand_example():
    # L = 1, H = 2, M = 3, N = 2.  Heads and question tokens are averaged (Eq. 1):
    #   head 0 rows (0.1, 0.1), (0.6, 0.0), (0.2, 0.4); head 1 rows (0.0, 0.3), (0.3, 0.3), (0.1, 0.1)
    #   column sums (1.3, 1.2) / 6 = (0.21667, 0.2)
    A = np.array([[[[0.1, 0.1], [0.6, 0.0], [0.2, 0.4]],
                   [[0.0, 0.3], [0.3, 0.3], [0.1, 0.1]]]])
    a = Q.aggregate_attention(A)
    np.testing.assert_allclose(a, [[1.3 / 6, 1.2 / 6]], rtol=1e-14)
    # l1 normalisation after averaging: (13/25, 12/25).  Normalising each row first
    # would give a different distribution, (0.5 + 1 + 1/3 + 0 + 0.5 + 0.5) / 6 = 0.4722 for token 0.
    np.testing.assert_allclose(Q.l1_normalise(a), [[13 / 25, 12 / 25]], rtol=1e-14)


def test_eq1_invariances():
    rng = np.random.default_rng(3)
    A = rng.random((3, 4, 5, 11))
    p = Q.l1_normalise(Q.aggregate_attention(A))
    np.testing.assert_allclose(p.sum(-1), 1.0, rtol=1e-14)
    # heads and question tokens are exchangeable
    np.testing.assert_allclose(Q.l1_normalise(Q.aggregate_attention(A[:, ::-1, rng.permutation(5)])), p, rtol=1e-13)
    # scale-free; visual-token permutations permute p
    np.testing.assert_allclose(Q.l1_normalise(Q.aggregate_attention(7.5 * A)), p, rtol=1e-13)
    perm = rng.permutation(11)
    np.testing.assert_allclose(Q.l1_normalise(Q.aggregate_attention(A[..., perm])), p[:, perm], rtol=1e-13)
    # rows that are full softmaxes over the visual tokens: the Eq. 1 average already sums to one
    S = rng.random((2, 3, 4, 6))
    S /= S.sum(-1, keepdims=True)
    np.testing.assert_allclose(Q.aggregate_attention(S).sum(-1), 1.0, rtol=1e-14)
    # rows that put all their attention on one token: a is the token frequency
    O = np.zeros((1, 2, 2, 4))
    O[0, 0, 0, 1] = O[0, 0, 1, 1] = O[0, 1, 0, 3] = 1.0
    O[0, 1, 1, 0] = 1.0
    np.testing.assert_allclose(Q.aggregate_attention(O), [[0.25, 0.5, 0.0, 0.25]])


def test_degenerate_layers_are_uniform():
    A = np.zeros((2, 3, 0, 5))        # no question tokens
    np.testing.assert_allclose(Q.l1_normalise(Q.aggregate_attention(A)), np.full((2, 5), 0.2))
    Z = np.zeros((1, 2, 2, 4))        # attention underflowed to zero
    np.testing.assert_allclose(Q.l1_normalise(Q.aggregate_attention(Z)), np.full((1, 4), 0.25))


def _js_point_mass_vs_uniform(N):
    # p = delta_0, q = 1/N: m_0 = (N+1)/(2N), m_n = 1/(2N)
    kl_p = math.log(2.0 * N / (N + 1))
    kl_q = (1.0 / N) * math.log(2.0 / (N + 1)) + (N - 1) / N * math.log(2.0)
    return 0.5 * (kl_p + kl_q)


def test_eq2_teacher_closed_form():
    N, H, M = 4, 2, 3
    ref = np.full((3, H, 2, N), 0.1)             # uniform reference attention in every layer
    A = np.full((3, H, M, N), 0.2)                # layer 0: uniform too -> JS = 0
    A[1] = 0.0
    A[1][..., :2] = 0.3                           # layer 1: uniform on half the tokens -> 3/4 ln(4/3)
    A[2] = 0.0
    A[2][..., 0] = 0.5                            # layer 2: a point mass
    r = Q.qcts(A, ref)
    np.testing.assert_allclose(r["js"], [0.0, 0.75 * math.log(4 / 3), _js_point_mass_vs_uniform(N)], atol=1e-15)
    assert r["layer"] == 2
    np.testing.assert_allclose(r["teacher"], [1, 0, 0, 0])
    np.testing.assert_allclose(r["p_ref"], 0.25)


def test_eq2_ties_go_to_the_lower_layer():
    rng = np.random.default_rng(4)
    A = np.repeat(rng.random((1, 2, 3, 8)), 4, axis=0)
    ref = np.repeat(rng.random((1, 2, 2, 8)), 4, axis=0)
    r = Q.qcts(A, ref)
    assert r["layer"] == 0
    assert Q.select_teacher_layer([0.1, 0.3, 0.3, 0.2]) == 1


def test_packed_batch_equals_single_samples():
    w = W.AttentionWorkload("tiny", 90, 3, 4, 3, 1, 6, 2, 9, 5)
    lens = np.array([4, 0, 7], np.int32)
    attn, lens, ref = W.make_attention_batch(w, lens=lens)
    assert attn.size == w.L * w.H * w.N * int(lens.sum())
    res = Q.qcts_batch(attn, lens, ref, w.L, w.H, w.N)
    for b in range(3):
        single = Q.qcts(Q.bf16_bits_to_f64(W.make_attention(w, b, int(lens[b]))),
                        Q.bf16_bits_to_f64(W.make_attention(w, b, w.m_ref, ref=True)))
        np.testing.assert_array_equal(res[b]["js"], single["js"])
        assert res[b]["layer"] == single["layer"]
    np.testing.assert_allclose(res[1]["p"], 1.0 / w.N)      # no question tokens: uniform


def test_synthetic_attention_has_a_middle_layer_teacher():
    # the generator's question pulls attention onto a region in the middle layers, so the
    # divergence is not flat and the teacher is a middle layer with a clear margin
    w = W.AttentionWorkload("mid", 91, 2, 16, 4, 1, 24, 8, 8, 7)
    attn, lens, ref = W.make_attention_batch(w)
    for r in Q.qcts_batch(attn, lens, ref, w.L, w.H, w.N):
        js = np.sort(r["js"])
        assert w.L // 8 <= r["layer"] <= w.L - w.L // 8
        assert (js[-1] - js[-2]) / js[-1] > 1e-3
        assert js[-1] > 5 * js[0]
