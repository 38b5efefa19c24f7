"""Pins of the parity rules and batch helpers that only the GPU tests call: the QCTS
teacher-layer rule (Eq. 2: the layer of largest divergence, ties to the lower layer), the
score and gradient error measures, the packed-attention split behind the batched QCTS
oracle, and the packed distillation batch (the loss is the mean over images of
D_KL(p* || p_hat)).  Each is held to hand-worked values or to a property that a
mistake in it breaks, not to a retyping of itself."""
import math

import numpy as np
import pytest

from oracle import distill_oracle as DO
from oracle import parity as P
from oracle import qcts_oracle as Q
from paper_2608_06411_gb300 import workloads as W


# ------------------------------------------------------------------ teacher-layer rule

def test_teacher_rule_takes_the_clear_maximum_only():
    js = np.array([0.10, 0.50, 0.20])            # margin (0.5 - 0.2) / 0.5 = 0.6, far above 1e-3
    assert P.check_teacher_layer(js, 1)[0]
    assert not P.check_teacher_layer(js, 2)[0]
    assert not P.check_teacher_layer(js, 0)[0]
    assert not P.check_teacher_layer(js, 3)[0]


def test_teacher_rule_accepts_either_layer_of_a_near_tie():
    js = np.array([0.5, 0.5 * (1 - 5e-4), 0.1])   # margin 5e-4 <= 1e-3: both top layers are valid
    assert P.check_teacher_layer(js, 0)[0]
    assert P.check_teacher_layer(js, 1)[0]
    assert not P.check_teacher_layer(js, 2)[0]     # far below the best
    assert not P.check_teacher_layer(js, -1)[0]    # out of range
    assert not P.check_teacher_layer(js, 3)[0]


def test_teacher_rule_margin_boundary():
    # just above the margin the lower-ranked layer is wrong; at a margin of 2e-3 it is rejected
    js = np.array([1.0, 1.0 - 2e-3])
    assert P.check_teacher_layer(js, 0)[0]
    assert not P.check_teacher_layer(js, 1)[0]
    assert P.check_teacher_layer(np.array([0.3]), 0)[0]    # a single layer


# ------------------------------------------------------------------ error measures

def test_score_relative_error_hand_values():
    p_ref = np.array([0.25, 0.5, 0.25])
    p_gpu = np.array([0.25, 0.5005, 0.2499], dtype=np.float32)
    # |0.0005| / 0.5 = 1e-3 and |0.0001| / 0.25 = 4e-4: the largest relative error is 1e-3
    assert P.score_rel_err(p_gpu, p_ref) == pytest.approx(1e-3, rel=1e-3)
    # relative, not absolute: a 1e-5 error on a score of 1e-4 is 0.1
    assert P.score_rel_err(np.array([1e-4 + 1e-5, 0.5]), np.array([1e-4, 0.5])) == pytest.approx(0.1, rel=1e-6)


def test_gradient_error_hand_values_and_scale_floor():
    g_ref = np.array([[2.0, -4.0], [1.0, 0.5]])
    g_gpu = g_ref + np.array([[0.0, 4e-4], [-1e-4, 0.0]])
    assert P.distill_grad_err(g_gpu, g_ref) == pytest.approx(1e-4, rel=1e-9)      # 4e-4 / max|g| = 4
    # a gradient that vanishes exactly is compared on the step's scale, not on itself
    assert P.distill_grad_err(np.full(3, 1e-8), np.zeros(3), scale=1e-3) == pytest.approx(1e-5, rel=1e-9)
    assert P.distill_grad_err(g_gpu, g_ref, scale=40.0) == pytest.approx(1e-5, rel=1e-9)


# ------------------------------------------------------------------ packed attention (QCTS batch)

def _blocks(lens, L=2, H=3, N=7, seed=0):
    rng = np.random.default_rng(seed)
    return [W.f32_to_bf16_bits(rng.gamma(1.0, size=(L, H, m, N)).astype(np.float32)) for m in lens]


def test_unpack_attention_recovers_each_sample_in_order():
    lens = [3, 0, 5, 1]                            # a sample without question tokens included
    blocks = _blocks(lens)
    packed = np.concatenate([b.reshape(-1) for b in blocks])
    out = Q.unpack_attention(packed, lens, 2, 3, 7)
    assert len(out) == len(lens)
    for b, (got, want) in enumerate(zip(out, blocks)):
        assert got.shape == (2, 3, lens[b], 7)
        np.testing.assert_array_equal(got, want)


def test_qcts_batch_is_per_sample_qcts():
    lens = [4, 2]
    blocks = _blocks(lens, seed=1)
    refs = np.stack(_blocks([3, 3], seed=2))
    packed = np.concatenate([b.reshape(-1) for b in blocks])
    res = Q.qcts_batch(packed, lens, refs, 2, 3, 7)
    for b in range(len(lens)):
        alone = Q.qcts(Q.bf16_bits_to_f64(blocks[b]), Q.bf16_bits_to_f64(refs[b]))
        np.testing.assert_array_equal(res[b]["js"], alone["js"])
        assert res[b]["layer"] == alone["layer"]


# ------------------------------------------------------------------ packed distillation batch

def _distill_inputs(seed=3, D=8, Dh=6, dp=4, N=5, lens=(3, 2)):
    rng = np.random.default_rng(seed)
    shapes = {"wT1": (Dh, D), "bT1": (Dh,), "wT2": (Dh, Dh), "bT2": (Dh,), "wQ": (dp, Dh),
              "wV1": (Dh, D), "bV1": (Dh,), "wV2": (Dh, Dh), "bV2": (Dh,), "wK": (dp, Dh)}
    wbits = {k: W.f32_to_bf16_bits((rng.standard_normal(s) / math.sqrt(s[-1])).astype(np.float32))
             for k, s in shapes.items()}
    text = W.f32_to_bf16_bits(rng.standard_normal((sum(lens), D)).astype(np.float32))
    vis = W.f32_to_bf16_bits(rng.standard_normal((len(lens), N, D)).astype(np.float32))
    t = rng.gamma(1.0, size=(len(lens), N))
    return text, vis, list(lens), t / t.sum(axis=1, keepdims=True), wbits


def test_distill_batch_is_the_mean_of_its_samples():
    text, vis, lens, teachers, wbits = _distill_inputs()
    loss, grads = DO.distill_batch(text, vis, lens, teachers, wbits)
    off = [0, lens[0], lens[0] + lens[1]]
    singles = [DO.distill_batch(text[off[b]:off[b + 1]], vis[b:b + 1], [lens[b]], teachers[b:b + 1], wbits)
               for b in range(2)]
    assert loss == pytest.approx(0.5 * (singles[0][0] + singles[1][0]), rel=1e-12)
    for k in DO.WEIGHT_NAMES:
        np.testing.assert_allclose(grads[k], 0.5 * (singles[0][1][k] + singles[1][1][k]), rtol=1e-10, atol=1e-14)


def test_distill_batch_pairs_each_question_with_its_own_image():
    # swapping the two images (with their teachers) but not the questions changes the loss:
    # the packed questions are matched to images by position
    text, vis, lens, teachers, wbits = _distill_inputs(lens=(3, 3))
    loss, _ = DO.distill_batch(text, vis, lens, teachers, wbits)
    swapped, _ = DO.distill_batch(text, vis[::-1].copy(), lens, teachers[::-1].copy(), wbits)
    assert abs(loss - swapped) > 1e-6 * abs(loss)
