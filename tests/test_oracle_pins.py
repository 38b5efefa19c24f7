"""Pins for the CPU oracle: each check ties it to something other than itself
(tabulated constants, closed forms, library routines, determinants, brute force,
invariants), so that a dropped term, a wrong sign or index or a transposed operand
in the oracle fails at least one of them.  CPU only.
"""
import itertools
import math

import numpy as np
import pytest
import scipy.special
import torch

from oracle import map_oracle as O
from oracle import parity as P
from paper_2608_06411_gb300 import workloads as W


def bits(x):
    return W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


# ------------------------------------------------------------------ storage (bf16)

def test_bf16_decode_known_patterns():
    pat = np.array([0x3F80, 0xC000, 0x3F00, 0x4049, 0x0001, 0x7F7F, 0x0000], dtype=np.uint16)
    want = [1.0, -2.0, 0.5, 3.140625, 2.0 ** -133, 3.3895313892515355e38, 0.0]
    assert O.bf16_bits_to_f64(pat).tolist() == want


# ------------------------------------------------------------------- predictor parts

def test_gelu_tabulated_values():
    # GELU(x) = x * Phi(x); Phi(1), Phi(2) from the standard normal table
    phi1, phi2 = 0.8413447460685429, 0.9772498680518208
    g = O.gelu(np.array([0.0, 1.0, -1.0, 2.0, -2.0]))
    np.testing.assert_allclose(g, [0.0, phi1, phi1 - 1.0, 2 * phi2, -2 * (1 - phi2)], rtol=1e-15, atol=1e-16)
    x = np.linspace(-5, 5, 101)
    np.testing.assert_allclose(O.gelu(x) - O.gelu(-x), x, atol=1e-14)


def _eye_bits(n, m=None):
    return bits(np.eye(n, m))


def test_mlp_is_exact_permutation_with_shifted_identity():
    # W1 = I, b1 = 16 keeps GELU in its linear regime (Phi(12) rounds to 1 in float64)
    # for integer inputs in [-4, 4]; W2 = P (a 3-cycle, so P != P^T), b2 = -16.
    # Then f(x) = P x exactly.
    n = 6
    P = np.zeros((n, n)); P[[0, 1, 2, 3, 4, 5], [1, 2, 0, 3, 5, 4]] = 1.0
    x = np.array([[-4, -1, 0, 1, 3, 4], [2, 2, -3, 0, 1, -2]], dtype=np.float64)
    w1, b1 = O.bf16_bits_to_f64(_eye_bits(n)), np.full(n, 16.0)
    w2, b2 = O.bf16_bits_to_f64(bits(P)), np.full(n, -16.0)
    out = O.mlp(x, w1, b1, w2, b2)
    np.testing.assert_array_equal(out, x @ P.T)
    assert not np.array_equal(out, x @ P)                 # the transposed operand differs


def test_mlp_keeps_hidden_activations_unrounded():
    # identity layers: f(x) = GELU(x) exactly, with no bf16 rounding of the hidden values
    x = np.array([[1.0, -1.0, 2.0, 0.5]])
    eye = np.eye(4)
    out = O.mlp(x, eye, np.zeros(4), eye, np.zeros(4))
    phi = [0.8413447460685429, 0.15865525393145707, 0.9772498680518208, 0.6914624612740131]
    want = [1.0 * phi[0], -1.0 * phi[1], 2.0 * phi[2], 0.5 * phi[3]]
    np.testing.assert_allclose(out[0], want, rtol=1e-15)


def test_mlp_second_layer_sees_exact_gelu():
    # layer 2 takes a difference of two GELU outputs: 1.0078125 Phi(1.0078125) - Phi(1)
    x = np.array([[1.0, 1.0078125]])
    w2 = np.array([[-1.0, 1.0], [0.0, 1.0]])
    out = O.mlp(x, np.eye(2), np.zeros(2), w2, np.zeros(2))
    g = x[0] * scipy.special.ndtr(x[0])
    np.testing.assert_allclose(out[0], [g[1] - g[0], g[1]], rtol=1e-13)


def test_mlp_nonsquare_selects_columns():
    # D = 6 -> Dh = 4 with W1[j, d] = 1 iff d == j + 2: layer 1 reads x[2:6]
    w1 = np.zeros((4, 6)); w1[np.arange(4), np.arange(4) + 2] = 1.0
    x = np.array([[9, 9, -1, 0, 2, 3]], dtype=np.float64)
    out = O.mlp(x, w1, np.full(4, 16.0), np.eye(4), np.full(4, -16.0))
    np.testing.assert_array_equal(out, [[-1, 0, 2, 3]])


def test_rope_single_pair_tabulated():
    c1, s1 = 0.5403023058681398, 0.8414709848078965       # cos 1, sin 1
    out = O.rope(np.array([[1.0, 0.0], [0.0, 1.0]]), np.array([1, 1]))
    np.testing.assert_allclose(out, [[c1, s1], [-s1, c1]], rtol=0, atol=1e-16)


def test_rope_pairs_are_half_apart_with_decaying_frequency():
    # d = 4: pairs (0, 2) at frequency 1 and (1, 3) at frequency 10000^(-1/2) = 0.01.
    c1, s1 = 0.5403023058681398, 0.8414709848078965
    out = O.rope(np.array([[0.0, 1.0, 0.0, 0.0]]), np.array([100]))
    np.testing.assert_allclose(out, [[0.0, c1, 0.0, s1]], atol=1e-15)
    out = O.rope(np.array([[1.0, 0.0, 0.0, 0.0]]), np.array([1]))
    np.testing.assert_allclose(out, [[c1, 0.0, s1, 0.0]], atol=1e-15)


def test_rope_inner_product_depends_on_offset_only():
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((1, 16)), rng.standard_normal((1, 16))
    for a, b in [(0, 5), (37, 42), (1000, 1005)]:
        lhs = (O.rope(q, np.array([a])) @ O.rope(k, np.array([b])).T).item()
        rhs = (q @ O.rope(k, np.array([b - a])).T).item()
        assert abs(lhs - rhs) < 1e-12


# --------------------------------------------------------------- predicted attention

def test_single_query_is_textbook_softmax():
    rng = np.random.default_rng(2)
    q, k = rng.standard_normal((1, 8)), rng.standard_normal((11, 8))
    want = scipy.special.softmax((q @ k.T)[0] / math.sqrt(8))
    np.testing.assert_allclose(O.predicted_attention(q, k), want, rtol=1e-14)


def test_two_tokens_is_logistic_of_scaled_gap():
    q = np.array([[1.0, -2.0, 0.5, 3.0]])
    k = np.array([[0.5, 1.0, -1.0, 2.0], [-1.0, 0.0, 2.0, 1.0]])
    gap = (q @ k[0] - q @ k[1]).item() / 2.0               # sqrt(d) = 2
    p = O.predicted_attention(q, k)
    np.testing.assert_allclose(p, [scipy.special.expit(gap), scipy.special.expit(-gap)], rtol=1e-14)


def test_mean_of_softmaxes_not_softmax_of_mean():
    # Eq. 3 averages M per-query softmaxes; closed form for this 2x3 case:
    # p = ((e+1)/(2(e+2)), (e+1)/(2(e+2)), 1/(e+2)).
    q = np.array([[2.0, 0, 0, 0], [0, 2.0, 0, 0]])
    k = np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0], [0, 0, 0, 0]])
    e = math.e
    want = [(e + 1) / (2 * (e + 2)), (e + 1) / (2 * (e + 2)), 1 / (e + 2)]
    p = O.predicted_attention(q, k)
    np.testing.assert_allclose(p, want, rtol=1e-14)
    other = scipy.special.softmax((q @ k.T).mean(0) / 2.0)
    assert np.abs(other - p).max() > 1e-2


def test_zero_key_projection_gives_uniform():
    dims = W.PredictorDims(D=32, Dh=16, dp=8)
    w = W.make_weights(dims, seed=3)
    w["wK"] = np.zeros_like(w["wK"])
    rng = np.random.default_rng(3)
    vis = bits(rng.standard_normal((1, 10, 32)))
    txt = bits(rng.standard_normal((4, 32)))
    p = O.map_score(txt, vis, [4], w)
    np.testing.assert_array_equal(p, np.full((1, 10), 1 / 10))


def _tiny_predictor_weights():
    """D = Dh = dp = 4: f_T, f_V are exact identities on small integers, W_Q = W_K = I."""
    eye = _eye_bits(4)
    return dict(wT1=eye, bT1=bits(np.full(4, 16.0)), wT2=eye, bT2=bits(np.full(4, -16.0)), wQ=eye,
                wV1=eye, bV1=bits(np.full(4, 16.0)), wV2=eye, bV2=bits(np.full(4, -16.0)), wK=eye)


def test_full_predictor_closed_form_without_rope():
    w = _tiny_predictor_weights()
    txt = bits([[2, 0, 0, 0], [0, 2, 0, 0]])
    vis = bits([[[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 0, 0]]])
    e = math.e
    want = [(e + 1) / (2 * (e + 2)), (e + 1) / (2 * (e + 2)), 1 / (e + 2)]
    np.testing.assert_allclose(O.map_score(txt, vis, [2], w, rope_on=False)[0], want, rtol=1e-14)


def test_full_predictor_closed_form_with_rope():
    # positions: visual n = 0, 1, 2; question m at N + m = 3, 4.  With d = 4 the pairs are
    # (0, 2) at frequency 1 and (1, 3) at frequency 0.01, and <R(a)x, R(b)y> = <x, R(b-a)y>:
    # logits / 2: m=0 -> (cos 3, 0, 0); m=1 -> (0, cos 0.03, 0).
    w = _tiny_predictor_weights()
    txt = bits([[2, 0, 0, 0], [0, 2, 0, 0]])
    vis = bits([[[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 0, 0]]])
    a, b = math.exp(math.cos(3.0)), math.exp(math.cos(0.03))
    s0 = np.array([a, 1.0, 1.0]) / (a + 2)
    s1 = np.array([1.0, b, 1.0]) / (b + 2)
    np.testing.assert_allclose(O.map_score(txt, vis, [2], w, rope_on=True)[0], (s0 + s1) / 2, rtol=1e-13)


def test_scores_are_a_distribution_and_shift_invariant():
    dims = W.PredictorDims(D=64, Dh=32, dp=16)
    w = W.make_weights(dims, seed=5, bias_std=0.1)
    rng = np.random.default_rng(5)
    vis, txt = bits(rng.standard_normal((20, 64))), bits(rng.standard_normal((6, 64)))
    q = O.predict_queries(txt, 20, w)
    k = O.predict_keys(vis, w)
    p = O.predicted_attention(q, k)
    assert abs(p.sum() - 1.0) < 1e-12 and (p > 0).all()
    q2 = O.predict_queries(txt, 20, w, pos=20 + np.arange(6) + 1234)
    k2 = O.predict_keys(vis, w, pos=np.arange(20) + 1234)
    np.testing.assert_allclose(O.predicted_attention(q2, k2), p, rtol=1e-9)


def test_scores_permutation_equivariant_with_positions():
    dims = W.PredictorDims(D=64, Dh=32, dp=16)
    w = W.make_weights(dims, seed=6)
    rng = np.random.default_rng(6)
    vis, txt = bits(rng.standard_normal((24, 64))), bits(rng.standard_normal((5, 64)))
    perm = rng.permutation(24)
    q = O.predict_queries(txt, 24, w)
    p = O.predicted_attention(q, O.predict_keys(vis, w))
    p_perm = O.predicted_attention(q, O.predict_keys(vis[perm], w, pos=perm))
    np.testing.assert_allclose(p_perm, p[perm], rtol=1e-12)
    # without RoPE, permuting the tokens alone permutes the scores
    q0 = O.predict_queries(txt, 24, w, rope_on=False)
    p0 = O.predicted_attention(q0, O.predict_keys(vis, w, rope_on=False))
    p0p = O.predicted_attention(q0, O.predict_keys(vis[perm], w, rope_on=False))
    np.testing.assert_allclose(p0p, p0[perm], rtol=1e-12)


def test_batch_equals_single_images():
    dims = W.PredictorDims(D=64, Dh=32, dp=16)
    w = W.make_weights(dims, seed=8)
    rng = np.random.default_rng(8)
    vis = bits(rng.standard_normal((3, 12, 64)))
    lens = [2, 5, 1]
    txt = bits(rng.standard_normal((8, 64)))
    p = O.map_score(txt, vis, lens, w)
    off = 0
    for b in range(3):
        np.testing.assert_array_equal(p[b], O.map_score(txt[off:off + lens[b]], vis[b:b + 1], [lens[b]], w)[0])
        off += lens[b]


def test_default_weights_give_nonuniform_scores():
    # guard against vacuous index-parity checks: logit std of the seeded init on a
    # small LLaVA-like case must be well above 0.5
    wl = W.WORKLOADS["c0"]
    dims = W.PredictorDims(D=wl.D, Dh=256, dp=128)
    w = W.make_weights(dims)
    vis = W.make_image(wl, 0)[:96]
    txt = W.make_text(wl, 0, 8)
    q = O.predict_queries(txt, 96, w)
    k = O.predict_keys(vis, w)
    assert ((q @ k.T) / math.sqrt(128)).std() > 0.5


# ------------------------------------------------------------------------- selection

def _sorted_topk(p, K):
    return sorted(range(len(p)), key=lambda i: (-p[i], i))[:K]


def test_zero_diversity_weight_is_topk():
    rng = np.random.default_rng(10)
    p = rng.dirichlet(np.ones(40))
    p[[3, 7, 11]] = p[5]                                   # ties go to the lower index
    V = rng.standard_normal((40, 16))
    for K0 in (0, 3, 10):
        r = O.select(p, V, 10, K0, lam=0.0)
        assert r["picks"].tolist() == _sorted_topk(p, 10)


def test_k0_equal_k_is_topk():
    rng = np.random.default_rng(11)
    p = rng.dirichlet(np.ones(30))
    V = rng.standard_normal((30, 8))
    assert O.select(p, V, 7, 7, lam=1.0)["picks"].tolist() == _sorted_topk(p, 7)


def test_k_at_least_n_keeps_everything():
    p = np.array([0.1, 0.5, 0.4])
    r = O.select(p, np.eye(3), 5, 2)
    assert r["keep"].tolist() == [0, 1, 2]


def _logdet(V, S):
    if not S:
        return 0.0
    sign, ld = np.linalg.slogdet(V[list(S)] @ V[list(S)].T)
    return ld if sign > 0 else -np.inf


def _objective(p, V, S, lam):
    # F(S) = sum log p_i + (lam / 2) log det G_S   (G = V V^T)
    return sum(math.log(p[i]) for i in S) + 0.5 * lam * _logdet(V, S)


@pytest.mark.parametrize("seed,N,K,K0,lam", [(0, 8, 4, 1, 1.0), (1, 10, 5, 2, 1.0), (2, 9, 6, 0, 0.5),
                                             (3, 12, 5, 2, 2.0), (4, 7, 3, 0, 1.0)])
def test_greedy_steps_against_determinants(seed, N, K, K0, lam):
    """Each greedy pick maximises the marginal gain of F computed from determinants
    (r_i^2 = det G_{S+i} / det G_S), an LU route independent of Gram-Schmidt.  Greedy
    never beats the brute-force optimum over K-subsets that contain R0."""
    rng = np.random.default_rng(seed)
    V = rng.standard_normal((N, 16))
    p = rng.dirichlet(np.ones(N))
    r = O.select(p, V, K, K0, lam=lam, tau=0.0)
    picks = r["picks"].tolist()
    S = picks[:K0]
    assert sorted(S) == sorted(_sorted_topk(p, K0))
    for j in picks[K0:]:
        gains = {i: math.log(p[i]) + 0.5 * lam * (_logdet(V, S + [i]) - _logdet(V, S))
                 for i in range(N) if i not in S}
        assert gains[j] >= max(gains.values()) - 1e-9
        S.append(j)
    f_greedy = _objective(p, V, picks, lam)
    rest = [i for i in range(N) if i not in picks[:K0]]
    f_opt = max(_objective(p, V, picks[:K0] + list(c), lam)
                for c in itertools.combinations(rest, K - K0))
    assert f_greedy <= f_opt + 1e-9
    assert f_greedy >= f_opt - 0.5 * abs(f_opt) - 5.0      # greedy is close to optimal


def test_orthogonal_tokens_greedy_equals_optimum():
    # with orthogonal embeddings residuals never shrink: greedy = top-K of p * ||v||^lam
    # = the brute-force optimum
    rng = np.random.default_rng(12)
    N, K, K0 = 9, 4, 1
    V = np.diag(rng.uniform(0.5, 2.0, N))
    p = rng.dirichlet(np.ones(N))
    for lam in (0.5, 1.0, 2.0):
        r = O.select(p, V, K, K0, lam=lam)
        r0 = _sorted_topk(p, K0)
        val = p * np.linalg.norm(V, axis=1) ** lam
        rest = sorted((i for i in range(N) if i not in r0), key=lambda i: (-val[i], i))[:K - K0]
        assert r["picks"].tolist() == r0 + rest
        best = max(itertools.combinations([i for i in range(N) if i not in r0], K - K0),
                   key=lambda c: _objective(p, V, r0 + list(c), lam))
        assert sorted(best) == sorted(rest)


def test_residuals_equal_determinant_ratios():
    rng = np.random.default_rng(13)
    V = rng.standard_normal((10, 12))
    b = O._Basis(V, tau=0.0)
    S = []
    for j in [4, 1, 7, 2]:
        b.add(j)
        S.append(j)
        r2 = b.r2()
        for i in range(10):
            if i in S:
                assert r2[i] < 1e-20
            else:
                want = math.exp(_logdet(V, S + [i]) - _logdet(V, S))
                assert abs(r2[i] - want) < 1e-10 * max(1.0, want)


def test_greedy_matches_gram_space_cholesky():
    """An independent algorithm for Eq. 4: pivoted incremental Cholesky on the Gram
    matrix G = V V^T (no D-space vectors) must pick the same tokens."""
    rng = np.random.default_rng(14)
    N, D, K, K0 = 200, 48, 40, 10
    cent = rng.standard_normal((20, D))
    V = cent[rng.integers(0, 20, N)] + 0.3 * rng.standard_normal((N, D))
    p = rng.dirichlet(np.ones(N) * 0.5)
    G = V @ V.T
    d2 = np.diag(G).copy()
    E = np.zeros((K, N))
    picks = list(_sorted_topk(p, K0))
    alive = np.ones(N, bool)
    t = 0

    def take(j):
        nonlocal t
        alive[j] = False
        e = (G[j] - E[:t, j] @ E[:t]) / math.sqrt(d2[j])
        E[t] = e
        d2[:] = d2 - e * e
        t += 1

    for j in picks:
        take(j)
    while len(picks) < K:
        val = np.where(alive, p * np.sqrt(np.maximum(d2, 0.0)), -np.inf)
        j = int(np.argmax(val))
        picks.append(j)
        take(j)
    r = O.select(p, V, K, K0, lam=1.0)
    assert r["picks"].tolist() == picks


def test_selection_invariants():
    rng = np.random.default_rng(15)
    N, D, K = 60, 24, 12
    V = rng.standard_normal((N, D))
    p = rng.dirichlet(np.ones(N))
    r = O.select(p, V, K, 4)
    keep = r["keep"]
    assert len(np.unique(keep)) == K and (np.diff(keep) > 0).all() and keep.min() >= 0 and keep.max() < N
    assert set(_sorted_topk(p, 4)) <= set(keep.tolist())
    assert O.select(3.0 * p, V, K, 4)["picks"].tolist() == r["picks"].tolist()
    assert O.select(p, 0.25 * V, K, 4)["picks"].tolist() == r["picks"].tolist()
    perm = rng.permutation(N)
    rp = O.select(p[perm], V[perm], K, 4)
    assert perm[rp["picks"]].tolist() == r["picks"].tolist()


def test_identical_tokens_have_zero_value_and_lowest_index_wins():
    e1, e2, e3 = np.eye(3)
    V = np.stack([e1, e1, e1, e2, e3, e1])
    p = np.array([0.3, 0.25, 0.2, 0.1, 0.1, 0.05])
    r = O.select(p, V, 5, 1)
    # R0 = {0}; copies of e1 now have value 0; 3 and 4 tie at 0.1 -> 3 first; then 4;
    # then all remaining are 0 -> lowest index 1
    assert r["picks"].tolist() == [0, 3, 4, 1, 2]
    assert r["basis"] == 3


def test_replay_of_own_picks_agrees_everywhere():
    rng = np.random.default_rng(16)
    V = rng.standard_normal((50, 20))
    p = rng.dirichlet(np.ones(50))
    r = O.select(p, V, 15, 5)
    rep = O.select_replay(p, V, 15, 5, r["picks"])
    assert all(s["forced"] == s["best"] for s in rep["steps"])
    assert rep["r0"].tolist() == r["picks"][:5].tolist()


def test_gather_copies_rows():
    rng = np.random.default_rng(17)
    vis = rng.integers(0, 2 ** 16, size=(2, 9, 5), dtype=np.uint16)
    keep = np.array([[0, 4, 8], [1, 2, 3]])
    out = O.gather(vis, keep)
    for b in range(2):
        for j in range(3):
            assert (out[b, j] == vis[b, keep[b, j]]).all()


def test_near_duplicate_pick_does_not_extend_basis():
    # v1 = e1 + 1e-3 e2 has ||residual||^2 / ||v1||^2 ~ 1e-6 <= tau after v0 = e1, so it is
    # kept (it is in R0) but adds no direction; e2 then still has residual 1 and wins.
    e1, e2, e3 = np.eye(3)
    V = np.stack([e1, e1 + 1e-3 * e2, e2, e3])
    p = np.array([0.4, 0.3, 0.2, 0.1])
    r = O.select(p, V, 3, 2, tau=1e-5)
    assert r["picks"].tolist() == [0, 1, 2] and r["basis"] == 2
    # with no threshold the noise direction enters the basis and e2 loses its residual
    assert O.select(p, V, 3, 2, tau=0.0)["picks"].tolist() == [0, 1, 3]


def test_r0_ties_go_to_lower_index():
    p = np.array([0.1, 0.3, 0.1, 0.3, 0.2])
    r = O.select(p, np.eye(5), 3, 3)
    assert r["picks"].tolist() == [1, 3, 4]
    assert O.select(p, np.eye(5), 4, 4)["picks"].tolist() == [1, 3, 4, 0]


def test_assemble_hand_example():
    # B = 2 images of N = 4 tokens (D = 2), k = 2 kept each, question lengths 1 and 2.
    # Image 0 keeps tokens 1, 3 then its question token; image 1 keeps 0, 2 then two tokens.
    vis = np.arange(16, dtype=np.uint16).reshape(2, 4, 2)
    text = np.array([[100, 101], [200, 201], [300, 301]], dtype=np.uint16)
    seq, pos = O.assemble(vis, np.array([[1, 3], [0, 2]]), text, [1, 2], pos_offset=5)
    np.testing.assert_array_equal(seq, [[2, 3], [6, 7], [100, 101],
                                        [8, 9], [12, 13], [200, 201], [300, 301]])
    # kept tokens keep their original positions; question tokens follow the whole image (N + m)
    np.testing.assert_array_equal(pos, [6, 8, 9, 5, 7, 9, 10])
    # ragged batch: image 1 has 3 valid tokens, so its question starts at position 3
    _, pos = O.assemble(vis, np.array([[1, 3], [0, 2]]), text, [1, 2], n_valid=[4, 3])
    np.testing.assert_array_equal(pos, [1, 3, 4, 0, 2, 3, 4])
    # an image without question tokens contributes its kept tokens only; k = 0 leaves the questions
    seq, pos = O.assemble(vis, np.zeros((2, 0), np.int64), text, [3, 0])
    np.testing.assert_array_equal(seq, text)
    np.testing.assert_array_equal(pos, [4, 5, 6])


# ------------------------------------------------------------------ the forced-replay parity checker
# The GPU selection is accepted by oracle/parity.py::check_selection: a pick must be the
# oracle's argmax wherever the oracle's margin (v1 - v2) / v1 exceeds 1e-4; below that margin
# any near-best token is valid and the check continues from it.  These cases feed the checker
# pick orders that did not come from the oracle, built by hand on orthogonal tokens whose
# values p_i * ||residual_i|| are known in closed form.

def _orthogonal_case():
    """Eight orthonormal tokens, value_i = p_i at every step.  K0 = 1, K = 6.  Greedy order
    by p: 0 (R0), 1, 2, then 4 (0.100004) over 3 (0.1) with margin 4e-5 (below 1e-4), 7, 5."""
    p = np.array([0.30, 0.20, 0.15, 0.10, 0.100004, 0.05, 0.04, 0.056])
    return p, np.eye(8), 6, 1


def test_checker_accepts_the_oracle_order_and_counts_its_near_tie():
    p, V, K, K0 = _orthogonal_case()
    order = [0, 1, 2, 4, 3, 7]
    assert O.select(p, V, K, K0)["picks"].tolist() == order
    rep = P.check_selection(p, V, K, K0, order, sorted(order))
    assert rep["ok"] and rep["identical"] and rep["sub_margin_steps"] == 1


def test_checker_accepts_a_swap_below_the_margin():
    p, V, K, K0 = _orthogonal_case()
    rep = P.check_selection(p, V, K, K0, [0, 1, 2, 3, 4, 7], [0, 1, 2, 3, 4, 7])
    assert rep["ok"] and not rep["identical"] and rep["sub_margin_steps"] == 1


def test_checker_rejects_a_wrong_pick_above_the_margin():
    p, V, K, K0 = _orthogonal_case()
    rep = P.check_selection(p, V, K, K0, [0, 1, 7, 2, 4, 3], [0, 1, 2, 3, 4, 7])
    assert not rep["ok"] and "picked 7" in rep["reason"]
    # the same set in another order is still wrong: token 2 must come before 4 and 3
    assert not P.check_selection(p, V, K, K0, [0, 1, 4, 2, 3, 7])["ok"]


def test_checker_rejects_repeated_out_of_range_and_unsorted_picks():
    p, V, K, K0 = _orthogonal_case()
    assert not P.check_selection(p, V, K, K0, [0, 1, 2, 4, 4, 7])["ok"]
    assert not P.check_selection(p, V, K, K0, [0, 1, 2, 4, 3, 8])["ok"]
    assert not P.check_selection(p, V, K, K0, [0, 1, 2, 4, 3])["ok"]
    assert not P.check_selection(p, V, K, K0, [0, 1, 2, 4, 3, 7], [0, 1, 2, 3, 7, 4])["ok"]


def test_checker_rejects_a_wrong_r0():
    p, V, K, K0 = _orthogonal_case()
    # the top-1 set is {0}, with a wide boundary margin (0.30 vs 0.20)
    rep = P.check_selection(p, V, K, K0, [1, 0, 2, 4, 3, 7], [0, 1, 2, 3, 4, 7])
    assert not rep["ok"] and "R0" in rep["reason"]
    assert not P.check_selection(p, V, 6, 2, [0, 2, 1, 4, 3, 7])["ok"]     # R0 out of p order


def _divergent_case():
    """Tokens 0 = e1 and 1 = (cos .3, sin .3, 0, 0) tie below the margin (values 1 and
    0.99995).  After picking 0 the best next token is 2 = e2 (0.6 against 0.59 for 3 = e3);
    after picking 1 instead, e2 keeps a residual of cos .3, so 2 is worth 0.6 cos .3 = 0.573
    and 3 (0.59) wins.  Both paths are valid; they keep different sets."""
    t = 0.3
    V = np.array([[1.0, 0, 0, 0], [math.cos(t), math.sin(t), 0, 0], [0, 1.0, 0, 0], [0, 0, 1.0, 0]])
    p = np.array([1.0, 0.99995, 0.6, 0.59])
    return p, V, 2, 0


def test_checker_follows_the_gpu_path_after_a_near_tie():
    p, V, K, K0 = _divergent_case()
    assert O.select(p, V, K, K0)["picks"].tolist() == [0, 2]
    rep = P.check_selection(p, V, K, K0, [1, 3], [1, 3])
    assert rep["ok"] and rep["sub_margin_steps"] == 1 and not rep["identical"]
    # the replay evaluates step 1 with token 1 (not the oracle's 0) in the basis
    steps = O.select_replay(p, V, K, K0, [1, 3])["steps"]
    assert [s["best"] for s in steps] == [0, 3]
    assert abs(steps[1]["v_best"] - 0.59) < 1e-12
    # continuing from 1, token 2 is no longer the best: [1, 2] is a wrong pick above the margin
    assert not P.check_selection(p, V, K, K0, [1, 2])["ok"]
