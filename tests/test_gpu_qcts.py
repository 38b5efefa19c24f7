"""QCTS teacher selection on the GPU (map_qcts through the C ABI) against the CPU oracle
(section "Question Contrastive Teacher Selection", Eq. 1-2)."""
import numpy as np
import pytest
import torch

from oracle import parity as P
from oracle import qcts_oracle as Q
from paper_2608_06411_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mb():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2608_06411_gb300 import binding
    return binding


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).cuda()


def _run(mb, attn, lens, ref, L, H, N):
    out = mb.qcts(_dev(attn), lens, _dev(ref), L, H, N)
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in out]


def _compare(res, p, p_ref, js, teacher, teacher_p):
    for b, r in enumerate(res):
        np.testing.assert_allclose(p[b], r["p"], rtol=P.QCTS_P_RTOL, atol=1e-30)
        np.testing.assert_allclose(p_ref[b], r["p_ref"], rtol=P.QCTS_P_RTOL, atol=1e-30)
        np.testing.assert_allclose(js[b], r["js"], rtol=P.QCTS_JS_RTOL, atol=P.QCTS_JS_ATOL)
        ok, why = P.check_teacher_layer(r["js"], int(teacher[b]))
        assert ok, f"sample {b}: {why}"
        np.testing.assert_array_equal(teacher_p[b], p[b, int(teacher[b])])


# N = 576 takes the 16-byte path, 7290 the 4-byte path, 37 the 2-byte path; the column
# tiles end raggedly in each case
@pytest.mark.parametrize("N", [576, 7290, 37, 1000])
def test_qcts_matches_oracle(mb, N):
    w = W.AttentionWorkload("t", 92, 4, 5, 3, 1, 24, 1, 9, 3)
    lens = np.array([4, 0, 9, 1], np.int32)
    attn, lens, ref = W.make_attention_batch(w, lens=lens, N=N)
    p, p_ref, js, teacher, teacher_p = _run(mb, attn, lens, ref, w.L, w.H, N)
    res = Q.qcts_batch(attn, lens, ref, w.L, w.H, N)
    _compare(res, p, p_ref, js, teacher, teacher_p)
    np.testing.assert_array_equal(p[1], np.float32(1.0 / N))     # no question tokens: uniform


def test_qcts_edge_cases(mb):
    L, H, N, M = 3, 2, 64, 5
    rng = np.random.default_rng(5)
    A = W.f32_to_bf16_bits(rng.random((L, H, M, N), dtype=np.float32) * np.float32(0.01))
    A[1] = 0                                   # layer 1: attention underflowed to zero
    ref = A.copy()[None]                       # the same attention for both questions
    p, p_ref, js, teacher, teacher_p = _run(mb, A.reshape(-1), [M], ref, L, H, N)
    np.testing.assert_array_equal(p, p_ref)
    np.testing.assert_array_equal(js, 0.0)     # identical distributions: every layer ties ...
    assert teacher[0] == 0                     # ... and the lower layer wins
    np.testing.assert_array_equal(p[0, 1], np.float32(1.0 / N))
    # a single layer, a single head, a single reference token
    w = W.AttentionWorkload("t1", 93, 1, 1, 1, 1, 8, 3, 3, 1)
    attn, lens, ref = W.make_attention_batch(w)
    out = _run(mb, attn, lens, ref, 1, 1, w.N)
    _compare(Q.qcts_batch(attn, lens, ref, 1, 1, w.N), *out)
    assert out[3][0] == 0


def test_qcts_is_deterministic(mb):
    w = W.AttentionWorkload("t2", 94, 2, 4, 4, 5, 24, 30, 60, 7)
    attn, lens, ref = W.make_attention_batch(w)
    a = _run(mb, attn, lens, ref, w.L, w.H, w.N)
    b = _run(mb, attn, lens, ref, w.L, w.H, w.N)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


def test_qcts_llava_next_full_size(mb):
    # the bench workload: 2 samples, 32 layers x 32 heads, N = 2880, ragged questions
    w = W.ATTENTION_WORKLOADS["q1"]
    attn, lens, ref = W.make_attention_batch(w, threads=16)
    out = _run(mb, attn, lens, ref, w.L, w.H, w.N)
    res = Q.qcts_batch(attn, lens, ref, w.L, w.H, w.N)
    _compare(res, *out)


def test_qcts_many_layers_split_over_launches(mb):
    # gridDim.z = samples * L is capped, so 40000 layers run one sample per launch
    L, H, N = 40000, 1, 16
    rng = np.random.default_rng(6)
    lens = np.array([1, 2], np.int32)
    attn = W.f32_to_bf16_bits(rng.random(L * H * N * 3, dtype=np.float32))
    ref = W.f32_to_bf16_bits(rng.random((2, L, H, 1, N), dtype=np.float32))
    out = _run(mb, attn, lens, ref, L, H, N)
    _compare(Q.qcts_batch(attn, lens, ref, L, H, N), *out)
