"""Pins of the distillation oracle (section "Cross-Modal Attention Distillation"): the KL
loss and its gradients against central finite differences, torch.autograd in float64, the
predictor forward of the scoring oracle, and the zero-loss point p* = p_hat."""
import math

import numpy as np
import pytest
import torch

from oracle import distill_oracle as DO
from oracle import map_oracle as O
from paper_2608_06411_gb300 import workloads as W


def _tiny(seed=0, D=8, Dh=6, dp=4, N=5, Ms=(3, 2)):
    rng = np.random.default_rng(seed)
    Wt = {"wT1": rng.standard_normal((Dh, D)) / math.sqrt(D), "bT1": 0.1 * rng.standard_normal(Dh),
          "wT2": rng.standard_normal((Dh, Dh)) / math.sqrt(Dh), "bT2": 0.1 * rng.standard_normal(Dh),
          "wQ": rng.standard_normal((dp, Dh)), "wV1": rng.standard_normal((Dh, D)) / math.sqrt(D),
          "bV1": 0.1 * rng.standard_normal(Dh), "wV2": rng.standard_normal((Dh, Dh)) / math.sqrt(Dh),
          "bV2": 0.1 * rng.standard_normal(Dh), "wK": rng.standard_normal((dp, Dh))}
    texts = [rng.standard_normal((m, D)) for m in Ms]
    visions = [rng.standard_normal((N, D)) for _ in Ms]
    teachers = []
    for _ in Ms:
        t = rng.gamma(1.0, size=N)
        teachers.append(t / t.sum())
    return Wt, texts, visions, teachers


def test_gradients_match_central_finite_differences():
    Wt, texts, visions, teachers = _tiny()
    _, grads = DO.loss_and_grads(texts, visions, teachers, Wt)
    rng = np.random.default_rng(1)
    h = 1e-6
    for name in DO.WEIGHT_NAMES:
        for _ in range(4):
            idx = tuple(int(rng.integers(s)) for s in Wt[name].shape)
            Wp = {k: v.copy() for k, v in Wt.items()}
            Wm = {k: v.copy() for k, v in Wt.items()}
            Wp[name][idx] += h
            Wm[name][idx] -= h
            lp, _ = DO.loss_and_grads(texts, visions, teachers, Wp)
            lm, _ = DO.loss_and_grads(texts, visions, teachers, Wm)
            fd = (lp - lm) / (2 * h)
            assert grads[name][idx] == pytest.approx(fd, rel=1e-5, abs=1e-8), (name, idx)


def test_gradients_match_torch_autograd_float64():
    Wt, texts, visions, teachers = _tiny(seed=2)
    loss, grads = DO.loss_and_grads(texts, visions, teachers, Wt)
    P = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in Wt.items()}

    def rope(x, pos):
        d = x.shape[1]
        half = d // 2
        freq = 10000.0 ** (-2.0 * torch.arange(half, dtype=torch.float64) / d)
        ang = torch.tensor(pos, dtype=torch.float64)[:, None] * freq[None, :]
        x1, x2 = x[:, :half], x[:, half:]
        return torch.cat([x1 * torch.cos(ang) - x2 * torch.sin(ang), x2 * torch.cos(ang) + x1 * torch.sin(ang)], 1)

    def mlp(x, a):
        z = x @ P["w%s1" % a].T + P["b%s1" % a]
        return torch.nn.functional.gelu(z) @ P["w%s2" % a].T + P["b%s2" % a]

    total = 0.0
    for t, v, ps in zip(texts, visions, teachers):
        t_, v_ = torch.tensor(t), torch.tensor(v)
        q = rope(mlp(t_, "T") @ P["wQ"].T, len(v) + np.arange(len(t)))
        k = rope(mlp(v_, "V") @ P["wK"].T, np.arange(len(v)))
        p_hat = torch.softmax(q @ k.T / math.sqrt(q.shape[1]), dim=1).mean(0)
        total = total + torch.nn.functional.kl_div(p_hat.log(), torch.tensor(ps), reduction="sum") / len(texts)
    total.backward()
    assert float(total.detach()) == pytest.approx(loss, rel=1e-12)
    for name in DO.WEIGHT_NAMES:
        np.testing.assert_allclose(grads[name], P[name].grad.numpy(), rtol=1e-9, atol=1e-13)


def test_forward_is_the_scoring_oracle():
    dims = W.PredictorDims(D=64, Dh=32, dp=8)
    wbits = W.make_weights(dims, seed=3)
    wl = W.WORKLOADS["c0"]
    vis = W.make_image(wl, 0, N=40, D=64)
    text = W.make_text(wl, 0, 6, D=64)
    f = DO.forward_image(O.bf16_bits_to_f64(text), O.bf16_bits_to_f64(vis), DO.decode_weights(wbits))
    np.testing.assert_allclose(f["p_hat"], O.map_score(text, vis[None], [6], wbits)[0], rtol=1e-13)


def test_teacher_equal_to_prediction_has_zero_loss_and_gradient():
    Wt, texts, visions, _ = _tiny(seed=4)
    teachers = [DO.forward_image(t, v, Wt)["p_hat"] for t, v in zip(texts, visions)]
    loss, grads = DO.loss_and_grads(texts, visions, teachers, Wt)
    assert abs(loss) < 1e-14
    for name in DO.WEIGHT_NAMES:
        assert np.abs(grads[name]).max() < 1e-12, name


def test_kl_closed_form():
    # D_KL((1/2, 1/2, 0) || (1/4, 1/4, 1/2)) = ln 2; zero-probability teacher entries add nothing
    assert DO.kl_divergence(np.array([0.5, 0.5, 0.0]), np.array([0.25, 0.25, 0.5])) == pytest.approx(math.log(2))


def test_key_bias_gradient_vanishes_without_rope():
    # every row of the softmax sums to one, so sum_n dL/dl[m, n] = 0: a shift common to all
    # keys (the key MLP's output bias, seen through W_K) has zero gradient when no position
    # rotates the keys differently
    Wt, texts, visions, teachers = _tiny(seed=5)
    _, g_off = DO.loss_and_grads(texts, visions, teachers, Wt, rope_on=False)
    assert np.abs(g_off["bV2"]).max() <= 1e-12 * np.abs(g_off["wV2"]).max()
    _, g_on = DO.loss_and_grads(texts, visions, teachers, Wt, rope_on=True)
    assert np.abs(g_on["bV2"]).max() > 1e-6 * np.abs(g_on["wV2"]).max()
