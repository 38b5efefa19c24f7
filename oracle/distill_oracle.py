"""CPU oracle for MAP's predictor distillation step (arxiv 2608.06411).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or execute this
module: only the tests and the CPU-baseline arm of ``bench.py`` use it.  It shares no code
with the CUDA library.

Section "Cross-Modal Attention Distillation": the predictor is trained offline by
minimising D_KL(p^{l*} || p_hat), the divergence from the teacher distribution that QCTS
selected to the predicted attention of Eq. 3.  This module computes that loss for a batch
of images and its gradient with respect to every predictor weight, in float64, by the chain
rule written out step by step in the reverse order of the forward pass:

  forward  (per image; the same steps as oracle.map_oracle)
    z1 = X W1^T + b1,  h1 = GELU(z1),  h2 = h1 W2^T + b2       (f_T on T, f_V on V)
    q' = h2_T W_Q^T,   k' = h2_V W_K^T
    q = RoPE(q', N + m),  k = RoPE(k', n)
    l[m, n] = <q_m, k_n> / sqrt(d),  s[m, :] = softmax_n(l[m, :]),  p_hat = mean_m s[m, :]
    L_b = sum_n p*_n (log p*_n - log p_hat_n)    (0 log 0 = 0);  L = mean_b L_b
  backward
    dL/dp_hat_n = -p*_n / (B p_hat_n)
    dL/ds[m, n] = (dL/dp_hat_n) / M
    dL/dl[m, n] = s[m, n] (dL/ds[m, n] - sum_n' s[m, n'] dL/ds[m, n'])      (softmax)
    dq = dl k / sqrt(d),  dk = dl^T q / sqrt(d)
    dq' = RoPE^T(dq), dk' = RoPE^T(dk)        (the transpose of the rotation: angle -a)
    dW_Q = sum_m dq'_m h2_m^T,  dh2 = dq' W_Q      (likewise W_K)
    dW2 = dh2^T h1,  db2 = sum_rows dh2,  dh1 = dh2 W2
    dz1 = dh1 * GELU'(z1),  GELU'(x) = Phi(x) + x phi(x)
    dW1 = dz1^T X,  db1 = sum_rows dz1

Readings (also in the design notes): the batch loss is the mean of the images' divergences;
inputs and weights are bf16 values decoded exactly, everything else float64; the teacher
p* is any distribution over each image's visual tokens (from QCTS in the paper).

Pins live in tests/test_distill_pins.py: central finite differences, torch.autograd in
float64, and the zero-loss / zero-gradient case p* = p_hat.
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import erf as _erf

from . import map_oracle as O

__all__ = ["WEIGHT_NAMES", "decode_weights", "forward_image", "loss_and_grads", "distill_batch"]

WEIGHT_NAMES = ("wT1", "bT1", "wT2", "bT2", "wQ", "wV1", "bV1", "wV2", "bV2", "wK")


def decode_weights(weights_bits: dict) -> dict:
    """bf16 bit patterns -> float64 arrays (exact)."""
    return {k: O.bf16_bits_to_f64(weights_bits[k]) for k in WEIGHT_NAMES}


def _gelu_grad(x: np.ndarray) -> np.ndarray:
    """d/dx [x Phi(x)] = Phi(x) + x phi(x)."""
    Phi = 0.5 * (1.0 + _erf(x / math.sqrt(2.0)))
    phi = np.exp(-0.5 * x * x) / math.sqrt(2.0 * math.pi)
    return Phi + x * phi


def _rope_angles(pos: np.ndarray, d: int, base: float):
    half = d // 2
    freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * freq[None, :]
    return np.cos(ang), np.sin(ang)


def _rope_backward(dy: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    """Gradient through y = RoPE(x): x1' = dy1 cos + dy2 sin, x2' = dy2 cos - dy1 sin."""
    half = dy.shape[1] // 2
    c, s = _rope_angles(pos, dy.shape[1], base)
    d1, d2 = dy[:, :half], dy[:, half:]
    return np.concatenate([d1 * c + d2 * s, d2 * c - d1 * s], axis=1)


def _mlp_forward(x, w1, b1, w2, b2):
    z1 = x @ w1.T + b1
    h1 = O.gelu(z1)
    h2 = h1 @ w2.T + b2
    return z1, h1, h2


def forward_image(t: np.ndarray, v: np.ndarray, W: dict, rope_base: float = 10000.0, rope_on: bool = True) -> dict:
    """The predictor's forward pass for one image with every intermediate kept.
    t [M, D], v [N, D] float64; W float64 weights.  rope_on=False puts every token at
    position 0 (RoPE becomes the identity)."""
    M, N = t.shape[0], v.shape[0]
    z1t, h1t, h2t = _mlp_forward(t, W["wT1"], W["bT1"], W["wT2"], W["bT2"])
    z1v, h1v, h2v = _mlp_forward(v, W["wV1"], W["bV1"], W["wV2"], W["bV2"])
    qp = h2t @ W["wQ"].T
    kp = h2v @ W["wK"].T
    pos_q = N + np.arange(M) if rope_on else np.zeros(M)
    pos_k = np.arange(N) if rope_on else np.zeros(N)
    q = O.rope(qp, pos_q, rope_base)
    k = O.rope(kp, pos_k, rope_base)
    d = q.shape[1]
    logits = (q @ k.T) / math.sqrt(d)
    logits = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(logits)
    s = e / e.sum(axis=1, keepdims=True)
    p_hat = s.mean(axis=0)
    return dict(t=t, v=v, z1t=z1t, h1t=h1t, h2t=h2t, z1v=z1v, h1v=h1v, h2v=h2v, q=q, k=k, s=s, p_hat=p_hat,
                pos_q=pos_q, pos_k=pos_k)


def kl_divergence(p_star: np.ndarray, p_hat: np.ndarray) -> float:
    """D_KL(p* || p_hat) = sum_n p*_n log(p*_n / p_hat_n), with 0 log 0 = 0."""
    pos = p_star > 0
    return float(np.sum(np.where(pos, p_star * np.log(np.where(pos, p_star, 1.0) / p_hat), 0.0)))


def _mlp_backward(dh2, x, z1, h1, w2):
    dW2 = dh2.T @ h1
    db2 = dh2.sum(axis=0)
    dh1 = dh2 @ w2
    dz1 = dh1 * _gelu_grad(z1)
    dW1 = dz1.T @ x
    db1 = dz1.sum(axis=0)
    return dW1, db1, dW2, db2


def _softmax_mean_backward(s: np.ndarray, g: np.ndarray) -> np.ndarray:
    """dL/dl from dL/dp_hat = g, through p_hat = mean_m softmax_n(l[m, :]) (s = the softmax)."""
    M = s.shape[0]
    ds = np.broadcast_to(g / M, s.shape)                 # dL/ds
    return s * (ds - (s * ds).sum(axis=1, keepdims=True))


def _logits_backward(dl: np.ndarray, q: np.ndarray, k: np.ndarray):
    """(dq, dk) through l = q k^T / sqrt(d)."""
    d = q.shape[1]
    return dl @ k / math.sqrt(d), dl.T @ q / math.sqrt(d)


def _teacher_grad(p_star: np.ndarray, p_hat: np.ndarray, B: int) -> np.ndarray:
    """dL/dp_hat of L = (1/B) sum_b D_KL(p*_b || p_hat_b)."""
    return -p_star / (B * p_hat)


def loss_and_grads(texts: list, visions: list, teachers: list, W: dict, rope_base: float = 10000.0,
                   rope_on: bool = True):
    """Batch loss L = mean_b D_KL(p*_b || p_hat_b) and dL/dW for every weight.

    texts[b] [M_b, D], visions[b] [N, D], teachers[b] [N] (float64; each teacher sums to 1)."""
    B = len(texts)
    grads = {k: np.zeros_like(W[k]) for k in WEIGHT_NAMES}
    loss = 0.0
    for b in range(B):
        f = forward_image(texts[b], visions[b], W, rope_base, rope_on)
        p_star, p_hat, s = teachers[b], f["p_hat"], f["s"]
        loss += kl_divergence(p_star, p_hat) / B
        g = _teacher_grad(p_star, p_hat, B)
        dl = _softmax_mean_backward(s, g)
        dq, dk = _logits_backward(dl, f["q"], f["k"])
        dqp = _rope_backward(dq, f["pos_q"], rope_base)
        dkp = _rope_backward(dk, f["pos_k"], rope_base)
        grads["wQ"] += dqp.T @ f["h2t"]
        grads["wK"] += dkp.T @ f["h2v"]
        dh2t = dqp @ W["wQ"]
        dh2v = dkp @ W["wK"]
        dW1, db1, dW2, db2 = _mlp_backward(dh2t, f["t"], f["z1t"], f["h1t"], W["wT2"])
        grads["wT1"] += dW1
        grads["bT1"] += db1
        grads["wT2"] += dW2
        grads["bT2"] += db2
        dW1, db1, dW2, db2 = _mlp_backward(dh2v, f["v"], f["z1v"], f["h1v"], W["wV2"])
        grads["wV1"] += dW1
        grads["bV1"] += db1
        grads["wV2"] += dW2
        grads["bV2"] += db2
    return loss, grads


def distill_batch(text_bits: np.ndarray, vis_bits: np.ndarray, lens, teachers: np.ndarray, weights_bits: dict,
                  rope_base: float = 10000.0, rope_on: bool = True):
    """loss_and_grads on a packed bf16 batch: vis [B, N, D], text [sum(lens), D], teachers [B, N]."""
    W = decode_weights(weights_bits)
    off = np.concatenate([[0], np.cumsum(np.asarray(lens, dtype=np.int64))])
    texts = [O.bf16_bits_to_f64(text_bits[off[b]:off[b + 1]]) for b in range(len(lens))]
    visions = [O.bf16_bits_to_f64(vis_bits[b]) for b in range(len(lens))]
    return loss_and_grads(texts, visions, [np.asarray(t, dtype=np.float64) for t in teachers], W, rope_base, rope_on)
