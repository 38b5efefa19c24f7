"""CPU oracle for MAP's Question Contrastive Teacher Selection (arxiv 2608.06411).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or execute
this module: only the tests and the CPU-baseline arm of ``bench.py`` use it.  It shares
no code with the CUDA library; its inputs are the seeded arrays of
``paper_2608_06411_gb300.workloads`` (passed in by the caller) and explicit arguments.

Plain numpy in float64, one function per step, written to be checked against the paper
by eye.  Section "Question Contrastive Teacher Selection":
  * Eq. 1: a^l_n = 1/(H M) * sum_h sum_m A^l[h, m, n]  (text-to-vision attention of
    layer l averaged over heads and question tokens);
  * l1 normalisation over the visual tokens gives the target distribution p^l;
  * the same aggregation and normalisation of the reference question's attention gives
    p_ref^l;
  * Eq. 2: l* = argmax_l D_JS(p^l, p_ref^l); p^{l*} is the teacher distribution.

Readings where the paper is silent (each is also listed in the design notes):
  * D_JS(p, q) = KL(p || m)/2 + KL(q || m)/2 with m = (p + q)/2, natural logarithm,
    0 * log 0 = 0.  (The log base does not change the argmax.)
  * A layer whose aggregated attention sums to zero (no question tokens, or attention
    that underflowed to zero) has the uniform distribution 1/N.
  * Ties in Eq. 2 go to the lower layer index.
  * Inputs are bf16 attention probabilities (non-negative), decoded exactly.

Pins live in tests/test_qcts_pins.py (library routines, closed forms, hand-worked cases,
invariants).
"""
from __future__ import annotations

import numpy as np

__all__ = ["bf16_bits_to_f64", "aggregate_attention", "l1_normalise", "js_divergence",
           "select_teacher_layer", "qcts", "qcts_batch", "unpack_attention"]


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns exactly: a bf16 is the upper half of a float32."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def aggregate_attention(A: np.ndarray) -> np.ndarray:
    """Eq. 1: a[l, n] = (1 / (H M)) sum_h sum_m A[l, h, m, n] for A of shape [L, H, M, N].

    With M = 0 there is nothing to average; a is zero (and its distribution uniform)."""
    A = np.asarray(A, dtype=np.float64)
    L, H, M, N = A.shape
    if H * M == 0:
        return np.zeros((L, N))
    return A.sum(axis=(1, 2)) / (H * M)


def l1_normalise(a: np.ndarray) -> np.ndarray:
    """p[l] = a[l] / sum_n a[l, n] (the attention is non-negative, so this is the l1
    normalisation); a row that sums to zero becomes uniform."""
    a = np.asarray(a, dtype=np.float64)
    s = a.sum(axis=-1, keepdims=True)
    N = a.shape[-1]
    safe = np.where(s > 0, s, 1.0)
    return np.where(s > 0, a / safe, 1.0 / N)


def _kl(p: np.ndarray, q: np.ndarray) -> np.ndarray:
    """sum_n p_n log(p_n / q_n) over the last axis, with 0 log 0 = 0."""
    pos = p > 0
    ratio = np.where(pos, p, 1.0) / np.where(pos, q, 1.0)
    return np.where(pos, p * np.log(ratio), 0.0).sum(axis=-1)


def js_divergence(p: np.ndarray, q: np.ndarray) -> np.ndarray:
    """Jensen-Shannon divergence over the last axis (nats)."""
    p = np.asarray(p, dtype=np.float64)
    q = np.asarray(q, dtype=np.float64)
    m = 0.5 * (p + q)
    return 0.5 * _kl(p, m) + 0.5 * _kl(q, m)


def select_teacher_layer(js: np.ndarray) -> int:
    """Eq. 2: the layer with the largest divergence (np.argmax takes the first, i.e. the
    lower layer index, on ties)."""
    return int(np.argmax(np.asarray(js, dtype=np.float64)))


def qcts(A: np.ndarray, A_ref: np.ndarray) -> dict:
    """Teacher selection for one image/question pair.

    A [L, H, M, N] and A_ref [L, H, M_ref, N]: attention (float values) of the question's
    and of the reference question's tokens to the N visual tokens.
    Returns p, p_ref [L, N], js [L], layer l*, teacher = p[l*]."""
    p = l1_normalise(aggregate_attention(A))
    p_ref = l1_normalise(aggregate_attention(A_ref))
    js = js_divergence(p, p_ref)
    l_star = select_teacher_layer(js)
    return {"p": p, "p_ref": p_ref, "js": js, "layer": l_star, "teacher": p[l_star]}


def unpack_attention(attn_bits: np.ndarray, lens, L: int, H: int, N: int):
    """Splits the packed bf16 attention of a batch (samples' [L, H, M_b, N] blocks in
    sample order) into per-sample uint16 arrays."""
    out, o = [], 0
    for M in (int(x) for x in lens):
        n = L * H * M * N
        out.append(attn_bits[o:o + n].reshape(L, H, M, N))
        o += n
    return out


def qcts_batch(attn_bits: np.ndarray, lens, ref_bits: np.ndarray, L: int, H: int, N: int) -> list:
    """qcts() for every sample of a packed bf16 batch (see unpack_attention); ref_bits is
    [B, L, H, M_ref, N] bf16 bits."""
    blocks = unpack_attention(attn_bits, lens, L, H, N)
    return [qcts(bf16_bits_to_f64(blocks[b]), bf16_bits_to_f64(ref_bits[b])) for b in range(len(blocks))]
