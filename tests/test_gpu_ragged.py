"""Ragged batches (variable-resolution images in a padded layout, n_valid tokens per image)
through map_*_ragged against the CPU oracle run on each image's valid tokens alone."""
import numpy as np
import pytest
import torch

from oracle import map_oracle as O
from oracle import parity as P
from paper_2608_06411_gb300 import workloads as W

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_06411_gb300 import binding as mb  # noqa: E402

DEV = torch.device("cuda:0")


def dev_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def make_ctx(dims, **kw):
    w = W.make_weights(dims, seed=7)
    return mb.Context({k: dev_bits(v) for k, v in w.items()}, dims.D, dims.Dh, dims.dp, **kw), w


def _check_batch(ctx, w, vis, text, lens, nv, K, sample):
    vis_t, text_t = dev_bits(vis), dev_bits(text)
    p = ctx.score_ragged(text_t, vis_t, lens, nv)
    torch.cuda.synchronize()
    ctx.check()
    p_all = p.cpu().numpy().copy()
    off = np.concatenate([[0], np.cumsum(lens)])
    for b in range(len(nv)):
        assert np.all(p_all[b, nv[b]:] == 0.0), f"image {b}: padding has a score"
    for b in sample:
        ref = O.map_score(text[off[b]:off[b + 1]], vis[b:b + 1, :nv[b]], [lens[b]], w)[0]
        assert P.score_rel_err(p_all[b, :nv[b]], ref) <= 1e-3, f"image {b}"
        p_all[b, :nv[b]] = ref.astype(np.float32)      # both sides select on the oracle's scores
    keep, order = ctx.select_ragged(torch.from_numpy(p_all).to(DEV), vis_t, nv, K)
    torch.cuda.synchronize()
    ctx.check()
    keep, order = keep.cpu().numpy(), order.cpu().numpy()
    K0 = O.resolve_k0(K)
    for b in range(len(nv)):
        assert keep[b].max() < nv[b], f"image {b}: padding retained"
    for b in sample:
        rep = P.check_selection(p_all[b, :nv[b]].astype(np.float64), O.bf16_bits_to_f64(vis[b, :nv[b]]), K, K0,
                                order[b], keep[b])
        assert rep["ok"], f"image {b}: {rep['reason']}"
    return p_all, keep


def test_ragged_matches_oracle_per_image():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, w = make_ctx(dims)
    wl = W.RaggedWorkload("small", 95, 4, 300, 60, 512, 16, 0.3, 3, 40, 24)
    vis, text, lens, _ = W.make_ragged_batch(wl)
    nv = np.array([300, 150, 77, 233], np.int32)       # one image fills the padded length
    _, keep = _check_batch(ctx, w, vis, text, lens, nv, 24, sample=range(4))
    # hand-off: questions follow each image's own tokens
    seq, pos = ctx.assemble_ragged(dev_bits(vis), torch.from_numpy(keep).to(DEV), dev_bits(text), lens, nv, 5)
    torch.cuda.synchronize()
    ctx.check()
    s_ref, p_ref = O.assemble(vis, keep, text, lens, 5, n_valid=nv)
    np.testing.assert_array_equal(seq.cpu().numpy().view(np.uint16), s_ref)
    np.testing.assert_array_equal(pos.cpu().numpy(), p_ref)


def test_ragged_without_padding_equals_regular_path():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    wl = W.RaggedWorkload("full", 96, 3, 200, 60, 512, 16, 0.3, 5, 30, 20)
    vis, text, lens, _ = W.make_ragged_batch(wl)
    nv = np.full(3, 200, np.int32)
    vis_t, text_t = dev_bits(vis), dev_bits(text)
    pr = ctx.score_ragged(text_t, vis_t, lens, nv)
    p = ctx.score(text_t, vis_t, lens)
    kr, orr = ctx.select_ragged(pr, vis_t, nv, 20)
    k, o = ctx.select(p, vis_t, 20)
    torch.cuda.synchronize()
    ctx.check()
    np.testing.assert_array_equal(pr.cpu().numpy(), p.cpu().numpy())
    np.testing.assert_array_equal(kr.cpu().numpy(), k.cpu().numpy())
    np.testing.assert_array_equal(orr.cpu().numpy(), o.cpu().numpy())


def test_ragged_prune_host_buffers_equal_device_path():
    dims = W.PredictorDims(D=512, Dh=256, dp=64)
    ctx, _ = make_ctx(dims)
    wl = W.RaggedWorkload("prune", 97, 5, 256, 40, 512, 16, 0.3, 4, 25, 16)
    vis, text, lens, nv = W.make_ragged_batch(wl)
    B, N, K = vis.shape[0], vis.shape[1], 16
    out_h = np.zeros((B, K, dims.D), np.uint16)
    keep_h = np.zeros((B, K), np.int32)
    sc_h = np.zeros((B, N), np.float32)
    ctx.prune_ragged(text, vis, lens, nv, K, out_h, keep_h, sc_h)
    vis_t = dev_bits(vis)
    sc = ctx.score_ragged(dev_bits(text), vis_t, lens, nv)
    keep, _ = ctx.select_ragged(sc, vis_t, nv, K)
    out = ctx.gather(vis_t, keep)
    torch.cuda.synchronize()
    ctx.check()
    np.testing.assert_array_equal(sc_h, sc.cpu().numpy())
    np.testing.assert_array_equal(keep_h, keep.cpu().numpy())
    np.testing.assert_array_equal(out_h, out.cpu().numpy().view(np.uint16))


@pytest.mark.parametrize("K", [128, 512])
def test_ragged_qwen_config_sampled(K):
    """16 variable-resolution images of up to 1280 tokens (D = 3584), keep 128 or 512."""
    wl = W.RAGGED_WORKLOADS["c5"]
    ctx, w = make_ctx(W.PredictorDims(D=wl.D))
    vis, text, lens, nv = W.make_ragged_batch(wl, threads=8)
    assert nv.min() >= K
    _, keep = _check_batch(ctx, w, vis, text, lens, nv, K, sample=[int(np.argmin(nv)), int(np.argmax(nv))])
    out = ctx.gather(dev_bits(vis), torch.from_numpy(keep).to(DEV))
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy().view(np.uint16), O.gather(vis, keep))
