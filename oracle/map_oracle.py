"""CPU oracle for MAP's inference-time pruning path (arxiv 2608.06411).

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or execute
this module: only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline arm of
``bench.py`` use it.  It shares no code with the CUDA library; its only inputs are
the seeded arrays of ``paper_2608_06411_gb300.workloads`` (passed in by the caller)
and explicit arguments.

Plain, slow and written to be checked against the paper by eye: numpy in float64,
one function per step, a library matmul / sort / erf as the only primitives.

Steps and where the paper defines them
  * predictor, section "Cross-Modal Attention Distillation", Eq. 3:
      two modality MLPs f_T, f_V, query/key projections W_Q, W_K, RoPE on q and k,
      p_hat_n = (1/M) sum_m softmax_n(<W_Q f_T(t_m), W_K f_V(v_n)> / sqrt(d)).
  * pruning, section "Inference-Time Token Pruning", Eq. 4:
      R0 = top-K0 tokens by p_hat; B0 = orthonormalised {v_i : i in R0};
      i_t = argmax_{i in C_{t-1}} p_hat_i * ||v_i - B B^T v_i||_2;
      v_{i_t} is orthogonalised against B, normalised and appended; repeat to K;
      the kept tokens are restored to their original order.

Readings where the paper is silent (each is also listed in the design notes):
  * MLP = Linear -> GELU(erf) -> Linear with bias, width Dh; W_Q, W_K have no bias.
  * Precision: inputs and weights are bf16 (decoded exactly); everything computed
    from them is float64 with no intermediate rounding.  (Rounding the hidden MLP
    activations to bf16 would make two fp32-accumulating implementations of the same
    predictor disagree by ~3e-3 in p_hat at D = 4096, above the 1e-3 score tolerance.)
  * RoPE: rotate-half pairing (i, i + d/2), theta_i = base^(-2i/d), base 10000;
    visual token n sits at position n, question token m at position N + m.
  * The active Eq. 3 (mean of per-query softmaxes) is used, not the commented-out
    softmax-of-mean variant.
  * Diversity weight lambda: value_i = p_hat_i * rho_i ** lambda (lambda = 1 is Eq. 4,
    lambda = 0 is plain top-K), rho_i = ||residual_i|| unless ||residual_i||^2 <=
    tau * ||v_i||^2, where rho_i = 0 (a token already in the span adds nothing).
    A pick whose residual is that small is kept but does not extend the basis.
  * Ties go to the lower token index.  K >= N keeps every token.

Parity pins for every function here live in tests/test_oracle_pins.py and
tests/test_golden.py.  Parity unpinned: whether these random-init weights behave like
a trained predictor (needs the paper's weights and data, not available).
"""
from __future__ import annotations

import math

import numpy as np
from scipy.special import erf as _erf

__all__ = [
    "bf16_bits_to_f64", "gelu", "mlp", "rope", "predict_queries",
    "predict_keys", "predicted_attention", "map_score", "resolve_k0", "select",
    "select_replay", "gather", "assemble",
]


# ----------------------------------------------------------------------------- storage

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns exactly: a bf16 is the upper half of a float32."""
    b = np.asarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------- predictor

def gelu(x: np.ndarray) -> np.ndarray:
    """GELU(x) = x * Phi(x) = x/2 * (1 + erf(x / sqrt(2)))  (exact erf form)."""
    return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))


def mlp(x: np.ndarray, w1, b1, w2, b2) -> np.ndarray:
    """f(x) = Linear2(GELU(Linear1(x))).

    x [n, D] float64; w1 [Dh, D], w2 [Dh, Dh] (PyTorch [out, in] layout); b1, b2 [Dh].
    Section "Cross-Modal Attention Distillation": the modality-specific MLPs f_T, f_V.
    """
    h1 = gelu(x @ w1.T + b1)
    return h1 @ w2.T + b2


def rope(x: np.ndarray, pos: np.ndarray, base: float = 10000.0) -> np.ndarray:
    """Rotary position embedding, rotate-half convention.

    For pair (x_i, x_{i+d/2}) at position p with angle a = p * base**(-2i/d):
    (x_i cos a - x_{i+d/2} sin a,  x_{i+d/2} cos a + x_i sin a).
    """
    n, d = x.shape
    half = d // 2
    freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[:, :half], x[:, half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=1)


def _w(weights: dict, key: str) -> np.ndarray:
    return bf16_bits_to_f64(weights[key])


def predict_queries(text_bits: np.ndarray, N: int, weights: dict, rope_on: bool = True,
                    rope_base: float = 10000.0, pos: np.ndarray | None = None) -> np.ndarray:
    """q_m = RoPE(W_Q f_T(t_m), N + m) for the M question tokens of one image."""
    t = bf16_bits_to_f64(text_bits)
    h = mlp(t, _w(weights, "wT1"), _w(weights, "bT1"), _w(weights, "wT2"), _w(weights, "bT2"))
    q = h @ _w(weights, "wQ").T
    if rope_on:
        q = rope(q, N + np.arange(len(t)) if pos is None else pos, rope_base)
    return q


def predict_keys(vis_bits: np.ndarray, weights: dict, rope_on: bool = True,
                 rope_base: float = 10000.0, pos: np.ndarray | None = None) -> np.ndarray:
    """k_n = RoPE(W_K f_V(v_n), n) for the N visual tokens of one image."""
    v = bf16_bits_to_f64(vis_bits)
    h = mlp(v, _w(weights, "wV1"), _w(weights, "bV1"), _w(weights, "wV2"), _w(weights, "bV2"))
    k = h @ _w(weights, "wK").T
    if rope_on:
        k = rope(k, np.arange(len(v)) if pos is None else pos, rope_base)
    return k


def predicted_attention(q: np.ndarray, k: np.ndarray) -> np.ndarray:
    """Eq. 3: p_hat_n = (1/M) sum_m softmax_n(<q_m, k_n> / sqrt(d)), d = projection width.

    The softmax runs over the N visual tokens for each question token m; the M
    distributions are then averaged.
    """
    d = q.shape[1]
    logits = (q @ k.T) / math.sqrt(d)                 # [M, N]
    logits = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(logits)
    soft = e / e.sum(axis=1, keepdims=True)
    return soft.mean(axis=0)


def map_score(text_bits: np.ndarray, vis_bits: np.ndarray, lens, weights: dict,
              rope_on: bool = True, rope_base: float = 10000.0) -> np.ndarray:
    """p_hat [B, N] for a batch: vis_bits [B, N, D], text_bits packed [sum(lens), D]."""
    B, N, _ = vis_bits.shape
    out = np.empty((B, N), dtype=np.float64)
    off = 0
    for b in range(B):
        m = int(lens[b])
        q = predict_queries(text_bits[off:off + m], N, weights, rope_on, rope_base)
        k = predict_keys(vis_bits[b], weights, rope_on, rope_base)
        out[b] = predicted_attention(q, k)
        off += m
    return out


# ------------------------------------------------------------------------------ pruning

def resolve_k0(K: int, k0_frac: float = 0.5, k0_abs: int = -1) -> int:
    """|R0|: k0_abs if >= 0, else floor(k0_frac * K); clamped to [0, K]."""
    k0 = k0_abs if k0_abs >= 0 else int(math.floor(k0_frac * K))
    return max(0, min(K, k0))


class _Basis:
    """Orthonormal basis B of the retained embeddings, kept implicitly through the
    residuals of every token: residual_i = v_i - B B^T v_i (modified Gram-Schmidt)."""

    def __init__(self, V: np.ndarray, tau: float):
        self.res = np.array(V, dtype=np.float64, copy=True)
        self.sq = np.einsum("ij,ij->i", V, V)          # ||v_i||^2
        self.tau = tau
        self.size = 0

    def r2(self) -> np.ndarray:
        """||v_i - B B^T v_i||^2 for every token, from the residual vectors themselves."""
        return np.einsum("ij,ij->i", self.res, self.res)

    def rho(self) -> np.ndarray:
        r2 = self.r2()
        return np.where(r2 > self.tau * self.sq, np.sqrt(np.maximum(r2, 0.0)), 0.0)

    def add(self, j: int) -> bool:
        """Orthogonalise v_j against B (its residual), normalise, append; then remove the
        new direction from every token's residual.  Returns whether B grew."""
        rj = self.res[j].copy()
        r2j = float(rj @ rj)
        if not r2j > self.tau * self.sq[j]:
            return False
        b = rj / math.sqrt(r2j)
        self.res -= np.outer(self.res @ b, b)
        self.size += 1
        return True


def _values(p: np.ndarray, rho: np.ndarray, lam: float) -> np.ndarray:
    """value_i = p_hat_i * rho_i ** lambda; lambda = 0 gives p_hat itself."""
    if lam == 0.0:
        return p.astype(np.float64).copy()
    return p * rho ** lam


def _top_order(p: np.ndarray) -> np.ndarray:
    """Token indices by p_hat descending, ties to the lower index (a stable sort)."""
    return np.argsort(-np.asarray(p, dtype=np.float64), kind="stable")


def _margin(vals: np.ndarray) -> float:
    """Relative gap (v1 - v2) / v1 between the best and the runner-up value."""
    v = np.sort(vals[np.isfinite(vals)])[::-1]
    if len(v) < 2:
        return 1.0
    if v[0] <= 0.0:
        return 0.0
    return float((v[0] - v[1]) / v[0])


def select(p: np.ndarray, V: np.ndarray, K: int, K0: int, lam: float = 1.0,
           tau: float = 1e-5) -> dict:
    """Inference-time pruning (section "Inference-Time Token Pruning", Eq. 4).

    p [N] predicted attention, V [N, D] visual embeddings (float64; bf16 values decoded
    exactly).  Returns dict(picks = tokens in the order they were retained,
    keep = the same tokens restored to ascending original order, margins = relative
    gap between best and runner-up at each pick, basis = |B| at the end).
    """
    p = np.asarray(p, dtype=np.float64)
    N = len(p)
    if K >= N:
        idx = np.arange(N)
        return dict(picks=idx, keep=idx, margins=np.ones(N), basis=None)
    K0 = max(0, min(K0, K))
    order = _top_order(p)
    r0 = order[:K0]
    r0_margin = 1.0
    if 0 < K0 < N:
        a, b = p[order[K0 - 1]], p[order[K0]]
        r0_margin = float((a - b) / a) if a > 0 else 0.0
    basis = _Basis(V, tau)
    alive = np.ones(N, dtype=bool)
    picks, margins = [], []
    for j in r0:                                      # R0 and B0
        alive[j] = False
        picks.append(int(j)); margins.append(r0_margin)
        basis.add(int(j))
    while len(picks) < K:                             # greedy picks, Eq. 4
        vals = _values(p, basis.rho(), lam)
        vals[~alive] = -np.inf
        j = int(np.argmax(vals))                      # first maximum: lowest index
        margins.append(_margin(vals))
        alive[j] = False
        picks.append(j)
        basis.add(j)
    picks = np.array(picks, dtype=np.int64)
    return dict(picks=picks, keep=np.sort(picks), margins=np.array(margins),
                basis=basis.size)


def select_replay(p: np.ndarray, V: np.ndarray, K: int, K0: int, forced: np.ndarray,
                  lam: float = 1.0, tau: float = 1e-5) -> dict:
    """Replay a given pick order step by step (forced replay, for parity checks).

    At each greedy step the oracle evaluates every candidate, records its own argmax,
    the margin and the value of the forced pick, then continues from the forced pick.
    Returns dict(r0 = oracle R0 in order, steps = list of per-step dicts).
    """
    p = np.asarray(p, dtype=np.float64)
    N = len(p)
    K0 = max(0, min(K0, K))
    r0 = _top_order(p)[:K0]
    forced = [int(x) for x in forced]
    basis = _Basis(V, tau)
    alive = np.ones(N, dtype=bool)
    steps = []
    for t, j in enumerate(forced):
        if t < K0:
            alive[j] = False
            basis.add(j)
            continue
        vals = _values(p, basis.rho(), lam)
        vals[~alive] = -np.inf
        best = int(np.argmax(vals))
        steps.append(dict(t=t, forced=j, best=best, v_forced=float(vals[j]),
                          v_best=float(vals[best]), margin=_margin(vals),
                          forced_alive=bool(alive[j])))
        alive[j] = False
        basis.add(j)
    return dict(r0=r0, steps=steps)


def gather(vis_bits: np.ndarray, keep: np.ndarray) -> np.ndarray:
    """Compaction: out[b, j] = V[b, keep[b, j]] (a row copy of the bf16 bits)."""
    B = vis_bits.shape[0]
    return np.stack([vis_bits[b][np.asarray(keep[b], dtype=np.int64)] for b in range(B)])


def assemble(vis_bits: np.ndarray, keep: np.ndarray, text_bits: np.ndarray, lens, pos_offset: int = 0,
             n_valid=None):
    """Hand-off to the language model (section "Inference-Time Token Pruning", last
    paragraph): the kept tokens, restored to their original order, keep their positional
    indices and are combined with the question tokens.  Per image b: its k kept visual
    tokens (keep[b], ascending) at positions keep[b], then its M_b question tokens at
    positions N + m (the question follows the full image), all shifted by pos_offset;
    images one after another.  With n_valid (ragged batch: image b has n_valid[b] tokens,
    the rest of its rows are padding) the question follows the image's own tokens: N_b + m.
    Returns (seq [sum_b (k + M_b), D] bf16 bits, pos int32)."""
    B, N, _ = vis_bits.shape
    rows, pos = [], []
    o = 0
    for b in range(B):
        M = int(lens[b])
        Nb = N if n_valid is None else int(n_valid[b])
        rows.append(vis_bits[b][np.asarray(keep[b], dtype=np.int64)])
        rows.append(text_bits[o:o + M])
        pos.append(np.asarray(keep[b], dtype=np.int64) + pos_offset)
        pos.append(Nb + np.arange(M) + pos_offset)
        o += M
    return np.concatenate(rows, axis=0), np.concatenate(pos).astype(np.int32)
