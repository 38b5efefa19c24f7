"""GPU parity: the CUDA path through the C ABI against the CPU oracle (and, for the
GEMM building block, against a plain PyTorch fp32 reference).  Marked gpu."""
import numpy as np
import pytest
import torch

from oracle import map_oracle as O
from oracle import parity as P
from paper_2608_06411_gb300 import workloads as W

import _oracle_pool as OP

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_06411_gb300 import binding as mb  # noqa: E402

DEV = torch.device("cuda:0")


def dev_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def make_ctx(dims, seed=7, bias_std=0.0, **kw):
    w = W.make_weights(dims, seed=seed, bias_std=bias_std)
    return mb.Context({k: dev_bits(v) for k, v in w.items()}, dims.D, dims.Dh, dims.dp, **kw), w


def run_select(ctx, p32, vis, K):
    keep, order = ctx.select(torch.from_numpy(p32).to(DEV), dev_bits(vis), K)
    torch.cuda.synchronize()
    ctx.check()
    return keep.cpu().numpy(), order.cpu().numpy()


def assert_selection(p32, vis, K, K0, keep, order, lam=1.0, tau=1e-5, label=None):
    reps = []
    for b in range(len(p32)):
        rep = P.check_selection(p32[b].astype(np.float64), O.bf16_bits_to_f64(vis[b]), K, K0, order[b], keep[b],
                                lam=lam, tau=tau)
        assert rep["ok"], f"image {b}: {rep['reason']}"
        reps.append(rep)
    if label:
        OP.record(label, reps)


# ------------------------------------------------------------------ GEMM building block

@pytest.mark.parametrize("M,K,N", [(300, 512, 512), (128, 256, 192), (1, 64, 64), (1000, 1024, 256)])
@pytest.mark.parametrize("epi", [mb.EPI_GELU_BF16, mb.EPI_BIAS_BF16, mb.EPI_F32])
def test_linear_matches_torch_fp32(M, K, N, epi):
    ctx, _ = make_ctx(W.PredictorDims(D=256, Dh=256, dp=64))
    g = torch.Generator(device="cpu").manual_seed(M * 7 + N)
    x = torch.randn(M, K, generator=g).to(torch.bfloat16).to(DEV)
    w = (torch.randn(N, K, generator=g) / K ** 0.5).to(torch.bfloat16).to(DEV)
    b = torch.randn(N, generator=g).to(torch.bfloat16).to(DEV)
    y = ctx.linear(x, w, b, epi)
    torch.cuda.synchronize()
    ctx.check()
    ref = x.float() @ w.float().T
    if epi != mb.EPI_F32:
        ref = ref + b.float()
    if epi == mb.EPI_GELU_BF16:
        ref = torch.nn.functional.gelu(ref)
    if epi == mb.EPI_F32:
        err = (y - ref).abs().max().item()
        assert err <= 1e-4 * ref.abs().max().item() + 1e-5
    else:
        # bf16 outputs: at most one bf16 rounding step from the fp32 reference
        torch.testing.assert_close(y.float(), ref, rtol=2 ** -7, atol=1e-3)
        exact = (y == ref.to(torch.bfloat16)).float().mean().item()
        assert exact > 0.99


# ------------------------------------------------------------------ Eq. 3 scores

def test_scores_match_oracle_llava15_shape():
    wl = W.WORKLOADS["c0"]
    dims = W.PredictorDims()
    ctx, w = make_ctx(dims)
    vis = W.make_image(wl, 0)[None]
    lens = np.array([32], np.int32)
    text = W.make_text(wl, 0, 32)
    p, q, k = ctx.score_debug(dev_bits(text), dev_bits(vis), lens)
    torch.cuda.synchronize()
    ctx.check()
    q_ref = O.predict_queries(text, wl.N, w)
    k_ref = O.predict_keys(vis[0], w)
    assert np.linalg.norm(q.cpu().numpy() - q_ref) / np.linalg.norm(q_ref) < 2e-3
    assert np.linalg.norm(k.cpu().numpy() - k_ref) / np.linalg.norm(k_ref) < 2e-3
    p_ref = O.predicted_attention(q_ref, k_ref)
    assert P.score_rel_err(p.cpu().numpy()[0], p_ref) <= 1e-3


def test_scores_ragged_batch_with_biases():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, w = make_ctx(dims, seed=3, bias_std=0.1)
    wl = W.WORKLOADS["c1"]
    B, N = 3, 300
    lens = np.array([5, 130, 1], np.int32)
    vis = np.stack([W.make_image(wl, b, N=N, D=dims.D) for b in range(B)])
    text = np.concatenate([W.make_text(wl, b, int(lens[b]), D=dims.D) for b in range(B)])
    p = ctx.score(dev_bits(text), dev_bits(vis), lens)
    torch.cuda.synchronize()
    ctx.check()
    p_ref = O.map_score(text, vis, lens, w)
    assert P.score_rel_err(p.cpu().numpy(), p_ref) <= 1e-3
    np.testing.assert_allclose(p.cpu().numpy().sum(1), 1.0, atol=1e-5)


def test_scores_without_rope_are_permutation_equivariant():
    dims = W.PredictorDims(D=256, Dh=256, dp=128)
    ctx, w = make_ctx(dims, rope_on=False)
    wl = W.WORKLOADS["c0"]
    vis = W.make_image(wl, 1, N=257, D=dims.D)
    text = W.make_text(wl, 1, 7, D=dims.D)
    perm = np.random.default_rng(0).permutation(257)
    p1 = ctx.score(dev_bits(text), dev_bits(vis[None]), [7]).cpu().numpy()[0]
    p2 = ctx.score(dev_bits(text), dev_bits(vis[perm][None]), [7]).cpu().numpy()[0]
    ctx.check()
    # each token's key is computed alone; only the softmax sums see a different order
    np.testing.assert_allclose(p2, p1[perm], rtol=1e-6)
    p_ref = O.map_score(text, vis[None], [7], w, rope_on=False)[0]
    assert P.score_rel_err(p1, p_ref) <= 1e-3


# ------------------------------------------------------------------ Eq. 4 selection

def _oracle_scores(vis, lens, text, w, **kw):
    return O.map_score(text, vis, lens, w, **kw).astype(np.float32)


def test_select_matches_oracle_llava15_shape():
    wl = W.WORKLOADS["c0"]
    dims = W.PredictorDims()
    ctx, w = make_ctx(dims)
    vis = W.make_image(wl, 0)[None]
    text = W.make_text(wl, 0, 32)
    p32 = _oracle_scores(vis, [32], text, w)
    keep, order = run_select(ctx, p32, vis, wl.K)
    assert_selection(p32, vis, wl.K, O.resolve_k0(wl.K), keep, order, label="c0 N=576 k=32 (oracle scores)")


@pytest.mark.parametrize("lam,k0_frac,K", [(1.0, 0.0, 40), (1.0, 0.25, 64), (0.5, 0.5, 50), (2.0, 0.5, 33),
                                           (0.0, 0.5, 40), (1.0, 1.0, 40), (1.0, 0.5, 300), (1.0, 0.0, 200)])
def test_select_variants(lam, k0_frac, K):
    dims = W.PredictorDims(D=256, Dh=256, dp=64)
    ctx, _ = make_ctx(dims, lam=lam, k0_frac=k0_frac)
    wl = W.WORKLOADS["c1"]
    rng = np.random.default_rng(int(K + 100 * lam))
    B, N = 2, 700
    vis = np.stack([W.make_image(wl, b, N=N, D=dims.D) for b in range(B)])
    p32 = rng.dirichlet(np.full(N, 0.3), size=B).astype(np.float32)
    keep, order = run_select(ctx, p32, vis, K)
    assert_selection(p32, vis, K, O.resolve_k0(K, k0_frac), keep, order, lam=lam,
                     label=f"variants N=700 D=256 k={K} lambda={lam} K0={O.resolve_k0(K, k0_frac)}")


def test_select_duplicates_and_near_duplicates():
    dims = W.PredictorDims(D=256, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    rng = np.random.default_rng(5)
    N = 160
    base = rng.standard_normal((20, 256)).astype(np.float32)
    x = base[rng.integers(0, 20, N)]
    x[::3] += 1e-3 * rng.standard_normal((len(x[::3]), 256)).astype(np.float32)   # near-duplicates
    vis = W.f32_to_bf16_bits(x)[None]
    p32 = rng.dirichlet(np.ones(N), size=1).astype(np.float32)
    for K in (10, 40, 100):
        keep, order = run_select(ctx, p32, vis, K)
        assert_selection(p32, vis, K, O.resolve_k0(K), keep, order)


def test_select_edge_sizes():
    dims = W.PredictorDims(D=128, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    wl = W.WORKLOADS["c0"]
    N = 37
    vis = W.make_image(wl, 2, N=N, D=dims.D)[None]
    p32 = np.random.default_rng(1).dirichlet(np.ones(N), size=1).astype(np.float32)
    keep, order = run_select(ctx, p32, vis, N)
    assert keep.tolist() == [list(range(N))] and order.tolist() == [list(range(N))]
    for K in (1, 2, 36):
        keep, order = run_select(ctx, p32, vis, K)
        assert_selection(p32, vis, K, O.resolve_k0(K), keep, order)
    with pytest.raises(mb.MapError):
        ctx.select(torch.from_numpy(p32).to(DEV), dev_bits(vis), N + 1)
    k0, _ = ctx.select(torch.from_numpy(p32).to(DEV), dev_bits(vis), 0)
    assert k0.shape == (1, 0)


def test_select_batch_equals_single_images():
    dims = W.PredictorDims(D=256, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    wl = W.WORKLOADS["c3"]
    B, N, K = 5, 500, 60
    vis = np.stack([W.make_image(wl, b, N=N, D=dims.D) for b in range(B)])
    p32 = np.random.default_rng(2).dirichlet(np.full(N, 0.5), size=B).astype(np.float32)
    keep, order = run_select(ctx, p32, vis, K)
    for b in range(B):
        kb, ob = run_select(ctx, p32[b:b + 1], vis[b:b + 1], K)
        np.testing.assert_array_equal(ob[0], order[b])
        np.testing.assert_array_equal(kb[0], keep[b])


# ------------------------------------------------------------------ gather and the whole path

def test_gather_is_bit_exact():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    rng = np.random.default_rng(3)
    vis = rng.integers(0, 2 ** 16, size=(3, 90, 512), dtype=np.uint16)
    keep = np.sort(np.stack([rng.choice(90, 17, replace=False) for _ in range(3)]), 1).astype(np.int32)
    out = ctx.gather(dev_bits(vis), torch.from_numpy(keep).to(DEV))
    torch.cuda.synchronize()
    ctx.check()
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint16), O.gather(vis, keep))


def test_gather_rejects_bad_index_without_faulting():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    vis = torch.zeros((1, 10, 512), dtype=torch.int16, device=DEV)
    keep = torch.tensor([[0, 12]], dtype=torch.int32, device=DEV)
    ctx.gather(vis, keep)
    assert ctx.status() == mb.MAP_EINTERNAL
    assert ctx.status() == mb.MAP_OK


def test_assemble_is_bit_exact():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    rng = np.random.default_rng(4)
    B, N, K = 3, 90, 17
    vis = rng.integers(0, 2 ** 16, size=(B, N, 512), dtype=np.uint16)
    lens = np.array([5, 0, 12], np.int32)
    text = rng.integers(0, 2 ** 16, size=(int(lens.sum()), 512), dtype=np.uint16)
    keep = np.sort(np.stack([rng.choice(N, K, replace=False) for _ in range(B)]), 1).astype(np.int32)
    for k, off in [(K, 35), (0, 0), (N, 7)]:
        kp = keep[:, :k] if k <= K else np.tile(np.arange(N, dtype=np.int32), (B, 1))
        seq, pos = ctx.assemble(dev_bits(vis), torch.from_numpy(np.ascontiguousarray(kp)).to(DEV), dev_bits(text),
                                lens, pos_offset=off)
        torch.cuda.synchronize()
        ctx.check()
        s_ref, p_ref = O.assemble(vis, kp, text, lens, off)
        np.testing.assert_array_equal(seq.cpu().numpy().view(np.uint16), s_ref)
        np.testing.assert_array_equal(pos.cpu().numpy(), p_ref)


def test_assemble_many_images_split_over_launches():
    # image metadata travel as launch parameters, 512 images per launch
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    rng = np.random.default_rng(8)
    B, N, K = 1100, 6, 2
    vis = rng.integers(0, 2 ** 16, size=(B, N, 512), dtype=np.uint16)
    lens = rng.integers(0, 3, size=B).astype(np.int32)
    text = rng.integers(0, 2 ** 16, size=(int(lens.sum()), 512), dtype=np.uint16)
    keep = np.sort(np.stack([rng.choice(N, K, replace=False) for _ in range(B)]), 1).astype(np.int32)
    seq, pos = ctx.assemble(dev_bits(vis), torch.from_numpy(keep).to(DEV), dev_bits(text), lens, pos_offset=3)
    torch.cuda.synchronize()
    ctx.check()
    s_ref, p_ref = O.assemble(vis, keep, text, lens, 3)
    np.testing.assert_array_equal(seq.cpu().numpy().view(np.uint16), s_ref)
    np.testing.assert_array_equal(pos.cpu().numpy(), p_ref)


def test_assemble_rejects_bad_index_without_faulting():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    vis = torch.zeros((1, 10, 512), dtype=torch.int16, device=DEV)
    text = torch.ones((2, 512), dtype=torch.int16, device=DEV)
    keep = torch.tensor([[0, 12]], dtype=torch.int32, device=DEV)
    seq, pos = ctx.assemble(vis, keep, text, [2])
    assert ctx.status() == mb.MAP_EINTERNAL
    assert pos.cpu().tolist() == [0, -1, 10, 11]
    assert ctx.status() == mb.MAP_OK


def test_prune_host_buffers_equal_device_path():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, w = make_ctx(dims)
    wl = W.WORKLOADS["c1"]
    B, N, K = 5, 400, 30            # host buffers run as a pipeline of 4 image chunks (1, 1, 1, 2)
    lens = np.array([12, 40, 7, 33, 20], np.int32)
    vis = np.stack([W.make_image(wl, b, N=N, D=dims.D) for b in range(B)])
    text = np.concatenate([W.make_text(wl, b, int(lens[b]), D=dims.D) for b in range(B)])
    out_h = np.zeros((B, K, dims.D), np.uint16)
    keep_h = np.zeros((B, K), np.int32)
    sc_h = np.zeros((B, N), np.float32)
    ctx.prune(text, vis, lens, K, out_h, keep_h, sc_h)
    sc = ctx.score(dev_bits(text), dev_bits(vis), lens)
    keep, _ = ctx.select(sc, dev_bits(vis), K)
    out = ctx.gather(dev_bits(vis), keep)
    torch.cuda.synchronize()
    ctx.check()
    np.testing.assert_array_equal(sc_h, sc.cpu().numpy())
    np.testing.assert_array_equal(keep_h, keep.cpu().numpy())
    np.testing.assert_array_equal(out_h, out.cpu().numpy().view(np.uint16))
    assert P.score_rel_err(sc_h, O.map_score(text, vis, lens, w)) <= 1e-3


def test_llava_next_shape_end_to_end():
    """N = 2880, K = 160 (c1): scores against the oracle, then selection parity on the
    oracle's scores, then the gathered tokens bit for bit."""
    wl = W.WORKLOADS["c1"]
    dims = W.PredictorDims()
    ctx, w = make_ctx(dims)
    vis = W.make_image(wl, 0)[None]
    text = W.make_text(wl, 0, wl.m_lo)
    p = ctx.score(dev_bits(text), dev_bits(vis), [wl.m_lo])
    torch.cuda.synchronize()
    ctx.check()
    p_ref = O.map_score(text, vis, [wl.m_lo], w)
    assert P.score_rel_err(p.cpu().numpy(), p_ref) <= 1e-3
    p32 = p_ref.astype(np.float32)
    keep, order = run_select(ctx, p32, vis, wl.K)
    assert_selection(p32, vis, wl.K, O.resolve_k0(wl.K), keep, order, label="c1 N=2880 k=160 (oracle scores)")
    out = ctx.gather(dev_bits(vis), torch.from_numpy(keep).to(DEV))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint16), O.gather(vis, keep))


# ------------------------------------------------------------------ remaining workload configs

def _full_batch_parity(key, own_scores=False):
    """Every image of a batched configuration: GPU scores against the oracle (max relative
    error <= 1e-3), GPU selection on the oracle's scores checked by forced replay, gathered
    tokens and the hand-off sequence bit for bit.  With own_scores, map_prune's own GPU
    scores and pick order are checked against the oracle's greedy too (the product path as
    a user runs it).  The oracle runs in a pool of host processes."""
    wl = W.WORKLOADS[key]
    dims = W.PredictorDims(D=wl.D)
    ctx, w = make_ctx(dims)
    vis, text, lens = W.make_batch(wl, threads=8)
    B, N, K = wl.B, wl.N, wl.K
    K0 = O.resolve_k0(K)
    ex = OP.pool()
    f_scores = [ex.submit(OP.oracle_scores, key, b, int(lens[b])) for b in range(B)]
    vis_t, text_t = dev_bits(vis), dev_bits(text)
    # the product path: map_prune on device buffers, then its scores' pick order
    out_p = torch.empty((B, K, wl.D), dtype=torch.int16, device=DEV)
    keep_p = torch.empty((B, K), dtype=torch.int32, device=DEV)
    p_gpu_t = torch.empty((B, N), dtype=torch.float32, device=DEV)
    ctx.prune(text_t, vis_t, lens, K, out_p, keep_p, p_gpu_t)
    keep_s, order_s = ctx.select(p_gpu_t, vis_t, K)
    torch.cuda.synchronize()
    ctx.check()
    p_gpu = p_gpu_t.cpu().numpy()
    np.testing.assert_array_equal(keep_s.cpu().numpy(), keep_p.cpu().numpy())
    keep_pn = keep_p.cpu().numpy()
    np.testing.assert_array_equal(out_p.cpu().numpy().view(np.uint16), O.gather(vis, keep_pn))
    p_ref = np.stack([f.result() for f in f_scores])
    errs = [P.score_rel_err(p_gpu[b], p_ref[b]) for b in range(B)]
    assert max(errs) <= 1e-3, f"image {int(np.argmax(errs))}: score rel err {max(errs):.2e}"
    # both sides select on the oracle's scores rounded to fp32
    p32 = p_ref.astype(np.float32)
    keep, order = run_select(ctx, p32, vis, K)
    f_sel = [ex.submit(OP.oracle_check, key, b, p32[b], K, K0, order[b], keep[b]) for b in range(B)]
    order_sn = order_s.cpu().numpy()
    f_own = [ex.submit(OP.oracle_check, key, b, p_gpu[b], K, K0, order_sn[b], keep_pn[b])
             for b in range(B)] if own_scores else []
    out = ctx.gather(vis_t, torch.from_numpy(keep).to(DEV))
    seq, pos = ctx.assemble(vis_t, torch.from_numpy(keep).to(DEV), text_t, lens, pos_offset=35)
    torch.cuda.synchronize()
    ctx.check()
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint16), O.gather(vis, keep))
    s_ref, pos_ref = O.assemble(vis, keep, text, lens, 35)
    np.testing.assert_array_equal(seq.cpu().numpy().view(np.uint16), s_ref)
    np.testing.assert_array_equal(pos.cpu().numpy(), pos_ref)
    reps = [f.result() for f in f_sel]
    bad = [(b, r["reason"]) for b, r in enumerate(reps) if not r["ok"]]
    assert not bad, f"selection on the oracle's scores: {bad[:3]}"
    OP.record(f"{key} all {B} images (oracle scores)", reps, max(errs))
    if own_scores:
        reps = [f.result() for f in f_own]
        bad = [(b, r["reason"]) for b, r in enumerate(reps) if not r["ok"]]
        assert not bad, f"selection on the GPU's own scores: {bad[:3]}"
        OP.record(f"{key} all {B} images (map_prune's own GPU scores)", reps, max(errs))
    ctx.close()


def test_batched_serving_config_every_image():
    """64 images, N = 2880, k = 160, ragged questions, near-duplicate images (b % 10 == 0):
    every image, on the oracle's scores and on map_prune's own scores."""
    _full_batch_parity("c3", own_scores=True)


def test_high_token_config_every_image():
    """16 images, N = 7290, D = 3584, k = 405, questions up to 512 tokens (two column tiles
    in Eq. 3) and K0 = 202 (the projection pass on the first 128 R0 tokens, the other 74
    retained as forced picks in the next round; coordinates in global memory)."""
    assert W.make_lens(W.WORKLOADS["c4"]).max() > 256
    _full_batch_parity("c4")


_SWEEP = {}


def _sweep_inputs():
    if not _SWEEP:
        wl = W.WORKLOADS["c2"]
        w = W.make_weights(W.PredictorDims())
        vis = W.make_image(wl, 0)[None]
        text = W.make_text(wl, 0, wl.m_lo)
        _SWEEP["v"] = (vis, O.map_score(text, vis, [wl.m_lo], w).astype(np.float32))
    return _SWEEP["v"]


@pytest.mark.parametrize("K,lam,k0_frac", [(64, 1.0, 0.5), (128, 1.0, 0.5), (320, 1.0, 0.5), (640, 1.0, 0.5),
                                           (160, 0.0, 0.5), (160, 0.5, 0.5), (160, 2.0, 0.5),
                                           (160, 1.0, 0.0), (160, 1.0, 0.25), (160, 1.0, 1.0)])
def test_retention_sweep_config(K, lam, k0_frac):
    """N = 2880 LLaVA-NeXT image: retained budgets and diversity weights of the sweep."""
    wl = W.WORKLOADS["c2"]
    dims = W.PredictorDims()
    ctx, w = make_ctx(dims, lam=lam, k0_frac=k0_frac)
    vis, p32 = _sweep_inputs()
    keep, order = run_select(ctx, p32, vis, K)
    assert_selection(p32, vis, K, O.resolve_k0(K, k0_frac), keep, order, lam=lam,
                     label=f"c2 N=2880 k={K} lambda={lam} K0={O.resolve_k0(K, k0_frac)}")
