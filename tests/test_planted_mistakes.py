"""Planted-mistake sweep: each test plants one plausible mistake in an oracle (on the CPU,
by replacing one of its functions for the duration of the test) and requires that at least
one pin of that oracle then fails.  This shows the pins tie each oracle to the paper rather
than to itself: a dropped term, a wrong sign, index or axis, or a transposed operand is
caught.  CPU only."""
import inspect
import math

import numpy as np
import pytest

from oracle import distill_oracle as DO
from oracle import map_oracle as O
from oracle import parity as P
from oracle import qcts_oracle as Q

import test_distill_pins
import test_golden
import test_oracle_pins
import test_parity_rule_pins
import test_qcts_pins


def _some_pin_fails(*modules) -> bool:
    """Runs the modules' pin functions (every parameter set of a parametrized one) until one
    raises; True if one did."""
    for mod in modules:
        for name, fn in inspect.getmembers(mod, inspect.isfunction):
            if not name.startswith("test_") or fn.__module__ != mod.__name__:
                continue
            marks = [m for m in getattr(fn, "pytestmark", []) if m.name == "parametrize"]
            if marks:
                argnames, values = marks[0].args[0], marks[0].args[1]
                names = [a.strip() for a in argnames.split(",")] if isinstance(argnames, str) else list(argnames)
                calls = [dict(zip(names, v if len(names) > 1 else (v,))) for v in values]
            else:
                if inspect.signature(fn).parameters:
                    continue                        # needs a fixture: not a pure pin
                calls = [{}]
            for kw in calls:
                try:
                    fn(**kw)
                except Exception:
                    return True
    return False


def test_pins_pass_unmodified():
    assert not _some_pin_fails(test_oracle_pins, test_golden, test_qcts_pins, test_distill_pins,
                               test_parity_rule_pins)


# ------------------------------------------------------------------ scoring and selection oracle

def _rope_sign_flipped(x, pos, base=10000.0):
    n, d = x.shape
    half = d // 2
    freq = base ** (-2.0 * np.arange(half) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[:, :half], x[:, half:]
    return np.concatenate([x1 * c + x2 * s, x2 * c - x1 * s], axis=1)


def _rope_adjacent_pairs(x, pos, base=10000.0):
    n, d = x.shape
    freq = base ** (-2.0 * np.arange(d // 2) / d)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * freq[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[:, 0::2], x[:, 1::2]
    out = np.empty_like(x)
    out[:, 0::2] = x1 * c - x2 * s
    out[:, 1::2] = x2 * c + x1 * s
    return out


def _attention_unscaled(q, k):
    logits = q @ k.T
    logits = logits - logits.max(axis=1, keepdims=True)
    e = np.exp(logits)
    return (e / e.sum(axis=1, keepdims=True)).mean(axis=0)


def _attention_softmax_of_mean(q, k):
    logits = (q @ k.T).mean(axis=0) / math.sqrt(q.shape[1])
    e = np.exp(logits - logits.max())
    return e / e.sum()


def _mlp_without_gelu(x, w1, b1, w2, b2):
    return (x @ w1.T + b1) @ w2.T + b2


def _mlp_without_biases(x, w1, b1, w2, b2):
    return O.gelu(x @ w1.T) @ w2.T


def _top_order_ties_high(p):
    p = np.asarray(p, dtype=np.float64)
    order = np.argsort(-p[::-1], kind="stable")
    return (len(p) - 1 - order)


def _values_without_diversity(p, rho, lam):
    return p.astype(np.float64).copy()


def _add_without_update(self, j):
    rj = self.res[j]
    if not float(rj @ rj) > self.tau * self.sq[j]:
        return False
    self.size += 1
    return True


_orig_predict_queries = O.predict_queries


def _queries_at_own_positions(text_bits, N, weights, rope_on=True, rope_base=10000.0, pos=None):
    M = len(text_bits)
    return _orig_predict_queries(text_bits, N, weights, rope_on, rope_base, np.arange(M) if pos is None else pos)


@pytest.mark.parametrize("attr,bad", [
    ("rope", _rope_sign_flipped),
    ("rope", _rope_adjacent_pairs),
    ("predicted_attention", _attention_unscaled),
    ("predicted_attention", _attention_softmax_of_mean),
    ("mlp", _mlp_without_gelu),
    ("mlp", _mlp_without_biases),
    ("_top_order", _top_order_ties_high),
    ("_values", _values_without_diversity),
    ("predict_queries", _queries_at_own_positions),
])
def test_scoring_and_selection_mistakes_are_caught(monkeypatch, attr, bad):
    monkeypatch.setattr(O, attr, bad)
    assert _some_pin_fails(test_oracle_pins, test_golden)


def test_missing_basis_update_is_caught(monkeypatch):
    monkeypatch.setattr(O._Basis, "add", _add_without_update)
    assert _some_pin_fails(test_oracle_pins, test_golden)


# ------------------------------------------------------------------ the forced-replay checker

def _replay_from_own_best(p, V, K, K0, forced, lam=1.0, tau=1e-5):
    """select_replay that records the forced pick but continues from its own argmax."""
    p = np.asarray(p, dtype=np.float64)
    K0 = max(0, min(K0, K))
    basis = O._Basis(V, tau)
    alive = np.ones(len(p), dtype=bool)
    steps = []
    for t, j in enumerate(int(x) for x in forced):
        if t < K0:
            alive[j] = False
            basis.add(j)
            continue
        vals = O._values(p, basis.rho(), lam)
        vals[~alive] = -np.inf
        best = int(np.argmax(vals))
        steps.append(dict(t=t, forced=j, best=best, v_forced=float(vals[j]), v_best=float(vals[best]),
                          margin=O._margin(vals), forced_alive=bool(alive[j])))
        alive[best] = False
        basis.add(best)
    return dict(r0=O._top_order(p)[:K0], steps=steps)


def _checker_accepts_anything(p, V, K, K0, gpu_order, gpu_keep=None, lam=1.0, tau=1e-5, margin=1e-4):
    return dict(ok=True, reason="", sub_margin_steps=0, identical=True)


_orig_check_selection = P.check_selection


def _checker_without_r0(p, V, K, K0, gpu_order, gpu_keep=None, lam=1.0, tau=1e-5, margin=1e-4):
    return _orig_check_selection(p, V, K, 0, gpu_order, gpu_keep, lam, tau, margin)


def _checker_ignores_repeats(p, V, K, K0, gpu_order, gpu_keep=None, lam=1.0, tau=1e-5, margin=1e-4):
    order = list(dict.fromkeys(int(x) for x in np.asarray(gpu_order).reshape(-1)))
    if len(order) < K:
        return dict(ok=True, reason="", sub_margin_steps=0, identical=False)
    return _orig_check_selection(p, V, K, K0, order, None, lam, tau, margin)


def _checker_without_value_bound(p, V, K, K0, gpu_order, gpu_keep=None, lam=1.0, tau=1e-5, margin=1e-4):
    return _orig_check_selection(p, V, K, K0, gpu_order, gpu_keep, lam, tau, margin=1.0)


@pytest.mark.parametrize("target,attr,bad", [
    (O, "select_replay", _replay_from_own_best),
    (P, "check_selection", _checker_accepts_anything),
    (P, "check_selection", _checker_without_r0),
    (P, "check_selection", _checker_ignores_repeats),
    (P, "check_selection", _checker_without_value_bound),
])
def test_parity_checker_mistakes_are_caught(monkeypatch, target, attr, bad):
    monkeypatch.setattr(target, attr, bad)
    assert _some_pin_fails(test_oracle_pins)


# ------------------------------------------------------------------ QCTS oracle

def _js_without_halves(p, q):
    p = np.asarray(p, dtype=np.float64)
    q = np.asarray(q, dtype=np.float64)
    m = 0.5 * (p + q)
    return Q._kl(p, m) + Q._kl(q, m)


_orig_js = Q.js_divergence


def _js_log2(p, q):
    return _orig_js(p, q) / math.log(2.0)


def _aggregate_rows_normalised_first(A):
    A = np.asarray(A, dtype=np.float64)
    s = A.sum(axis=-1, keepdims=True)
    return (A / np.where(s > 0, s, 1.0)).mean(axis=(1, 2))


def _aggregate_first_head_only(A):
    A = np.asarray(A, dtype=np.float64)
    return A[:, 0].mean(axis=1)


def _teacher_argmin(js):
    return int(np.argmin(np.asarray(js, dtype=np.float64)))


def _teacher_ties_high(js):
    js = np.asarray(js, dtype=np.float64)
    return int(len(js) - 1 - np.argmax(js[::-1]))


@pytest.mark.filterwarnings("ignore::RuntimeWarning")
@pytest.mark.parametrize("attr,bad", [
    ("js_divergence", _js_without_halves),
    ("js_divergence", _js_log2),
    ("aggregate_attention", _aggregate_rows_normalised_first),
    ("aggregate_attention", _aggregate_first_head_only),
    ("select_teacher_layer", _teacher_argmin),
    ("select_teacher_layer", _teacher_ties_high),
])
def test_qcts_mistakes_are_caught(monkeypatch, attr, bad):
    monkeypatch.setattr(Q, attr, bad)
    assert _some_pin_fails(test_qcts_pins)


# ------------------------------------------------------------------ distillation oracle

def _softmax_back_without_centering(s, g):
    return s * np.broadcast_to(g / s.shape[0], s.shape)


def _logits_back_unscaled_keys(dl, q, k):
    return dl @ k / math.sqrt(q.shape[1]), dl.T @ q


def _teacher_grad_without_batch_mean(p_star, p_hat, B):
    return -p_star / p_hat


def _rope_back_forward_rotation(dy, pos, base):
    half = dy.shape[1] // 2
    c, s = DO._rope_angles(pos, dy.shape[1], base)
    d1, d2 = dy[:, :half], dy[:, half:]
    return np.concatenate([d1 * c - d2 * s, d2 * c + d1 * s], axis=1)


def _gelu_grad_phi_only(x):
    return 0.5 * (1.0 + np.vectorize(math.erf)(x / math.sqrt(2.0)))


_orig_mlp_backward = DO._mlp_backward


def _mlp_backward_mean_bias(dh2, x, z1, h1, w2):
    dW1, db1, dW2, db2 = _orig_mlp_backward(dh2, x, z1, h1, w2)
    return dW1, db1, dW2, db2 / dh2.shape[0]


@pytest.mark.parametrize("attr,bad", [
    ("_softmax_mean_backward", _softmax_back_without_centering),
    ("_logits_backward", _logits_back_unscaled_keys),
    ("_teacher_grad", _teacher_grad_without_batch_mean),
    ("_rope_backward", _rope_back_forward_rotation),
    ("_gelu_grad", _gelu_grad_phi_only),
    ("_mlp_backward", _mlp_backward_mean_bias),
])
def test_distillation_mistakes_are_caught(monkeypatch, attr, bad):
    monkeypatch.setattr(DO, attr, bad)
    assert _some_pin_fails(test_distill_pins)


# ------------------------------------------------------------------ parity rules and batch helpers

def _teacher_rule_accepts_anything(js_oracle, layer_gpu, margin=P.QCTS_LAYER_MARGIN):
    return True, ""


def _teacher_rule_argmax_only(js_oracle, layer_gpu, margin=P.QCTS_LAYER_MARGIN):
    ok = layer_gpu == int(np.argmax(np.asarray(js_oracle)))
    return ok, ""


def _score_err_absolute(p_gpu, p_ref):
    return float(np.abs(np.asarray(p_gpu, dtype=np.float64) - p_ref).max())


def _grad_err_without_scale(g_gpu, g_ref, scale=0.0):
    g_ref = np.asarray(g_ref, dtype=np.float64)
    return float(np.abs(np.asarray(g_gpu, dtype=np.float64) - g_ref).max() / max(float(np.abs(g_ref).max()), 1e-300))


def _unpack_reversed(attn_bits, lens, L, H, N):
    out, o = [], 0
    for M in (int(x) for x in reversed(list(lens))):
        n = L * H * M * N
        out.append(attn_bits[o:o + n].reshape(L, H, M, N))
        o += n
    return out[::-1]


_orig_distill_batch = DO.distill_batch


def _distill_batch_first_question_only(text_bits, vis_bits, lens, teachers, weights_bits, rope_base=10000.0,
                                       rope_on=True):
    m0 = int(lens[0])
    text = np.concatenate([text_bits[:m0]] * len(lens))
    return _orig_distill_batch(text, vis_bits, [m0] * len(lens), teachers, weights_bits, rope_base, rope_on)


@pytest.mark.parametrize("target,attr,bad", [
    (P, "check_teacher_layer", _teacher_rule_accepts_anything),
    (P, "check_teacher_layer", _teacher_rule_argmax_only),
    (P, "score_rel_err", _score_err_absolute),
    (P, "distill_grad_err", _grad_err_without_scale),
    (Q, "unpack_attention", _unpack_reversed),
    (DO, "distill_batch", _distill_batch_first_question_only),
])
def test_parity_rule_and_batch_helper_mistakes_are_caught(monkeypatch, target, attr, bad):
    monkeypatch.setattr(target, attr, bad)
    assert _some_pin_fails(test_parity_rule_pins)


# ------------------------------------------------------------------ hand-off and compaction oracles

_orig_assemble = O.assemble


def _assemble_questions_at_m(vis_bits, keep, text_bits, lens, pos_offset=0, n_valid=None):
    seq, pos = _orig_assemble(vis_bits, keep, text_bits, lens, pos_offset, n_valid)
    N = vis_bits.shape[1]
    pos = pos.copy()
    k = np.asarray(keep).shape[1]
    o = 0
    for b in range(vis_bits.shape[0]):
        M = int(lens[b])
        Nb = N if n_valid is None else int(n_valid[b])
        pos[o + k:o + k + M] -= Nb                     # question token m at position m
        o += k + M
    return seq, pos


def _assemble_offset_on_kept_only(vis_bits, keep, text_bits, lens, pos_offset=0, n_valid=None):
    seq, pos = _orig_assemble(vis_bits, keep, text_bits, lens, 0, n_valid)
    pos = pos.copy()
    k = np.asarray(keep).shape[1]
    o = 0
    for b in range(vis_bits.shape[0]):
        pos[o:o + k] += pos_offset
        o += k + int(lens[b])
    return seq, pos


def _gather_from_first_image(vis_bits, keep):
    return np.stack([vis_bits[0][np.asarray(keep[b], dtype=np.int64)] for b in range(vis_bits.shape[0])])


@pytest.mark.parametrize("attr,bad", [
    ("assemble", _assemble_questions_at_m),
    ("assemble", _assemble_offset_on_kept_only),
    ("gather", _gather_from_first_image),
])
def test_handoff_and_gather_mistakes_are_caught(monkeypatch, attr, bad):
    monkeypatch.setattr(O, attr, bad)
    assert _some_pin_fails(test_oracle_pins)
