"""The seeded input generators: determinism, bf16 rounding, clustered structure."""
import numpy as np
import torch

from paper_2608_06411_gb300 import workloads as W


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(100_000) * 10.0 ** rng.uniform(-20, 20, 100_000)).astype(np.float32)
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)
    np.testing.assert_array_equal(W.bf16_bits_to_f32(ours), torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_generators_are_deterministic():
    w = W.WORKLOADS["c0"]
    np.testing.assert_array_equal(W.make_image(w, 3, N=50), W.make_image(w, 3, N=50))
    assert not np.array_equal(W.make_image(w, 3, N=50), W.make_image(w, 4, N=50))
    np.testing.assert_array_equal(W.make_weights(W.PredictorDims(64, 32, 8))["wK"],
                                  W.make_weights(W.PredictorDims(64, 32, 8))["wK"])


def test_clustered_structure():
    w = W.WORKLOADS["c0"]
    v = W.bf16_bits_to_f32(W.make_image(w, 0)).astype(np.float64)
    # token (0,0) and (0,1) share a 6x6 block; (0,0) and (0,6) do not
    same = np.linalg.norm(v[0] - v[1]) / np.linalg.norm(v[0])
    diff = np.linalg.norm(v[0] - v[6]) / np.linalg.norm(v[0])
    assert same < 0.5 < diff


def test_near_duplicate_images_repeat_crop_zero():
    w = W.WORKLOADS["c3"]
    v = W.bf16_bits_to_f32(W.make_image(w, 0)).astype(np.float64)   # image 0: near-duplicate
    c = 576
    rel = np.linalg.norm(v[c:2 * c] - v[:c]) / np.linalg.norm(v[:c])
    assert rel < 0.1
    lens = W.make_lens(w)
    assert lens.min() >= 16 and lens.max() <= 256 and len(lens) == 64


def test_attention_generator_rows_are_partial_distributions():
    w = W.AttentionWorkload("t", 80, 2, 6, 3, 2, 12, 4, 9, 5)
    a = W.bf16_bits_to_f32(W.make_attention(w, 0, 7)).astype(np.float64)
    assert a.shape == (6, 3, 7, w.N) and np.all(a >= 0)
    rows = a.sum(axis=-1)
    assert rows.min() > 0.04 and rows.max() < 0.51          # visual share U(0.05, 0.5), bf16-rounded
    np.testing.assert_array_equal(W.make_attention(w, 0, 7), W.make_attention(w, 0, 7, threads=1))
    assert not np.array_equal(W.make_attention(w, 0, 7), W.make_attention(w, 1, 7))
    attn, lens, ref = W.make_attention_batch(w)
    assert attn.size == w.L * w.H * w.N * int(lens.sum()) and ref.shape == (2, 6, 3, 5, w.N)
    assert lens.min() >= 4 and lens.max() <= 9


def test_ragged_generator_shapes_and_padding():
    w = W.RaggedWorkload("t", 81, 5, 300, 100, 64, 16, 0.3, 2, 9, 10)
    vis, text, lens, nv = W.make_ragged_batch(w)
    assert vis.shape == (5, 300, 64) and text.shape == (int(lens.sum()), 64)
    assert np.all(nv >= 20) and np.all(nv <= 300)
    v = W.bf16_bits_to_f32(vis).astype(np.float64)
    for b in range(5):
        # clustered tokens have norms near sqrt(D) (centroid N(0,1) + noise); padding N(0, 5^2) is far larger
        assert np.linalg.norm(v[b, :nv[b]], axis=1).mean() < 12
        if nv[b] < 300:
            assert np.linalg.norm(v[b, nv[b]:], axis=1).mean() > 30
    np.testing.assert_array_equal(W.make_ragged_batch(w)[0], vis)
