"""Parity rules between the CUDA path and the oracle (test infrastructure only).

Scores:     max_n |p_gpu - p_ref| / p_ref <= 1e-3.
Selection:  the GPU and the oracle get the SAME fp32 scores and bf16 embeddings (both
            produced on the CPU).  The oracle's own greedy run is the reference: at every
            pick whose oracle margin (v1 - v2) / v1 exceeds 1e-4 the GPU must take the
            oracle's token; where the margin is smaller either near-best token is valid,
            and the check continues from the GPU's choice (forced replay) requiring its
            value to be within a factor (1 - 1e-4) of the best.
Gather:     bit-exact.
"""
from __future__ import annotations

import numpy as np

from . import map_oracle as O


def score_rel_err(p_gpu: np.ndarray, p_ref: np.ndarray) -> float:
    p_gpu = np.asarray(p_gpu, dtype=np.float64)
    return float((np.abs(p_gpu - p_ref) / p_ref).max())


def check_selection(p: np.ndarray, V: np.ndarray, K: int, K0: int, gpu_order, gpu_keep=None, lam: float = 1.0,
                    tau: float = 1e-5, margin: float = 1e-4) -> dict:
    """Returns dict(ok, reason, sub_margin_steps, identical).  p must be the exact
    float32 scores the GPU received (as float64), V the decoded bf16 embeddings."""
    gpu_order = [int(x) for x in np.asarray(gpu_order).reshape(-1)]
    N = len(p)
    if len(gpu_order) != K or len(set(gpu_order)) != K or min(gpu_order) < 0 or max(gpu_order) >= N:
        return dict(ok=False, reason="pick list is not K distinct tokens in range", sub_margin_steps=0,
                    identical=False)
    if gpu_keep is not None:
        keep = [int(x) for x in np.asarray(gpu_keep).reshape(-1)]
        if keep != sorted(gpu_order):
            return dict(ok=False, reason="keep_idx is not the picks in ascending order", sub_margin_steps=0,
                        identical=False)
    ref = O.select(p, V, K, K0, lam=lam, tau=tau)
    if K >= N:
        same = gpu_order == list(range(N))
        return dict(ok=same, reason="" if same else "K >= N must keep all in order", sub_margin_steps=0,
                    identical=same)
    K0 = max(0, min(K0, K))
    # R0: the top-K0 set must match exactly unless the K0 boundary is itself a near-tie
    r0_ref = ref["picks"][:K0].tolist()
    if gpu_order[:K0] != r0_ref:
        if not (K0 > 0 and ref["margins"][0] <= margin and sorted(gpu_order[:K0]) != sorted(r0_ref)):
            return dict(ok=False, reason=f"R0 differs: {gpu_order[:K0][:8]}... vs {r0_ref[:8]}...",
                        sub_margin_steps=0, identical=False)
    identical = gpu_order == ref["picks"].tolist()
    if identical:
        subm = int((ref["margins"][K0:] <= margin).sum())
        return dict(ok=True, reason="", sub_margin_steps=subm, identical=True)
    rep = O.select_replay(p, V, K, K0, gpu_order, lam=lam, tau=tau)
    subm = 0
    for s in rep["steps"]:
        if not s["forced_alive"]:
            return dict(ok=False, reason=f"step {s['t']}: token {s['forced']} picked twice", sub_margin_steps=subm,
                        identical=False)
        if s["margin"] <= margin:
            subm += 1
            if s["v_forced"] < (1.0 - margin) * s["v_best"]:
                return dict(ok=False, reason=f"step {s['t']}: value {s['v_forced']:.6g} < best {s['v_best']:.6g}",
                            sub_margin_steps=subm, identical=False)
        elif s["forced"] != s["best"]:
            return dict(ok=False, reason=f"step {s['t']}: picked {s['forced']}, oracle {s['best']} "
                                         f"(margin {s['margin']:.2e})", sub_margin_steps=subm, identical=False)
    return dict(ok=True, reason="", sub_margin_steps=subm, identical=False)


# ----------------------------------------------------------------------------- QCTS
# Distributions p^l, p_ref^l: elementwise relative error <= 2e-5 (fp32 sums of positive
# bf16 values, about 1e-6 expected).  Divergences: relative error <= 1e-4 (plus 1e-7
# absolute for near-zero values).  Teacher layer: equal to the oracle's wherever the
# oracle's relative margin (js1 - js2) / js1 exceeds 1e-3; otherwise any layer whose
# oracle divergence is within that margin of the largest.
QCTS_P_RTOL, QCTS_JS_RTOL, QCTS_JS_ATOL, QCTS_LAYER_MARGIN = 2e-5, 1e-4, 1e-7, 1e-3


def check_teacher_layer(js_oracle: np.ndarray, layer_gpu: int, margin: float = QCTS_LAYER_MARGIN) -> tuple:
    """(ok, reason) for the GPU's teacher layer against the oracle's divergences."""
    js = np.asarray(js_oracle, dtype=np.float64)
    order = np.argsort(-js, kind="stable")
    top = js[order[0]]
    second = js[order[1]] if len(js) > 1 else -np.inf
    rel = (top - second) / top if top > 0 else 0.0
    if rel > margin:
        ok = layer_gpu == int(order[0])
        return ok, "" if ok else f"layer {layer_gpu}, oracle {int(order[0])} (margin {rel:.2e})"
    ok = 0 <= layer_gpu < len(js) and js[layer_gpu] >= (1.0 - margin) * top
    return ok, "" if ok else f"layer {layer_gpu} js {js[layer_gpu] if 0 <= layer_gpu < len(js) else None} vs {top}"


# ----------------------------------------------------------------------------- distillation
# Loss: relative error <= 1e-5.  Gradients (fp32 chain against float64): per weight tensor,
# max |g_gpu - g_ref| <= 1e-4 * max |g_ref| (sums over up to ~10^4 tokens of fp32 products
# err by ~sqrt(T) eps relative to the tensor's scale, ~5e-6; the softmax backward's
# g - c difference adds about as much).
DISTILL_LOSS_RTOL, DISTILL_GRAD_TOL = 1e-5, 1e-4


def distill_grad_err(g_gpu: np.ndarray, g_ref: np.ndarray, scale: float = 0.0) -> float:
    """max |g_gpu - g_ref| / max(max |g_ref|, scale).  A gradient that vanishes exactly (the
    key bias without RoPE: the softmax over visual tokens ignores a shift common to every key)
    is compared on `scale`, 1e-3 of the largest gradient of the step."""
    g_ref = np.asarray(g_ref, dtype=np.float64)
    den = max(float(np.abs(g_ref).max()), scale, 1e-300)
    return float(np.abs(np.asarray(g_gpu, dtype=np.float64) - g_ref).max() / den)
