"""map_select_noalloc through the C ABI: same picks as map_select, on two calls in a row,
and the oracle's greedy picks (forced-replay rule).

The allocation-free entry point is for callers that cannot allocate device memory while
they prune (a fixed device-memory budget, another framework's caching pool, a serving
path that must not stall on cudaMalloc / cudaFree); it carves its workspace from a static
device array instead.  This file is collected last on purpose."""
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


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def _ctx(D, **kw):
    dims = W.PredictorDims(D=D, Dh=256, dp=64)
    w = W.make_weights(dims)
    return mb.Context({k: _dev(v) for k, v in w.items()}, dims.D, dims.Dh, dims.dp, **kw)


@pytest.mark.parametrize("wl_name,B,K", [("c0", 1, 32), ("c1", 1, 160), ("c3", 2, 60)])
def test_noalloc_select_matches_map_select(wl_name, B, K):
    wl = W.WORKLOADS[wl_name]
    ctx = _ctx(wl.D)
    vis = np.stack([W.make_image(wl, b) for b in range(B)])
    rng = np.random.default_rng(B * 1000 + K)
    p_np = rng.dirichlet(np.full(wl.N, 0.3), size=B).astype(np.float32)
    p = torch.from_numpy(p_np).to(DEV)
    vis_t = _dev(vis)
    keep_ref, order_ref = ctx.select(p, vis_t, K)
    torch.cuda.synchronize()
    ctx.check()
    for _ in range(2):                       # two calls in a row share the static array
        keep = torch.full((B, K), -1, dtype=torch.int32, device=DEV)
        order = torch.full((B, K), -1, dtype=torch.int32, device=DEV)
        ctx.select_noalloc(p, vis_t, K, keep, order)
        torch.cuda.synchronize()
        ctx.check()
        assert torch.equal(keep, keep_ref) and torch.equal(order, order_ref)
    keep_np, order_np = keep.cpu().numpy(), order.cpu().numpy()
    for b in range(B):
        rep = P.check_selection(p_np[b].astype(np.float64), O.bf16_bits_to_f64(vis[b]), K, O.resolve_k0(K),
                                order_np[b], keep_np[b])
        assert rep["ok"], f"image {b}: {rep['reason']}"
    ctx.close()


def test_noalloc_plain_top_k_beyond_the_diversity_limit():
    """lambda = 0: plain top-k, allowed up to k = 4096 as in map_select."""
    wl = W.WORKLOADS["c1"]
    ctx = _ctx(wl.D, lam=0.0)
    N, K = 3000, 1500
    rng = np.random.default_rng(11)
    p_np = rng.dirichlet(np.full(N, 0.5), size=1).astype(np.float32)
    vis = torch.zeros((1, N, wl.D), dtype=torch.int16, device=DEV)
    p = torch.from_numpy(p_np).to(DEV)
    keep_ref, order_ref = ctx.select(p, vis, K)
    keep = torch.empty((1, K), dtype=torch.int32, device=DEV)
    order = torch.empty((1, K), dtype=torch.int32, device=DEV)
    ctx.select_noalloc(p, vis, K, keep, order)
    torch.cuda.synchronize()
    ctx.check()
    assert torch.equal(keep, keep_ref) and torch.equal(order, order_ref)
    np.testing.assert_array_equal(order.cpu().numpy()[0], np.argsort(-p_np[0].astype(np.float64), kind="stable")[:K])
    ctx.close()


def test_noalloc_select_rejects_oversized_workspace():
    wl = W.WORKLOADS["c1"]
    ctx = _ctx(wl.D)
    B = 8                                    # 8 LLaVA-NeXT images need ~46 MB > 16 MiB
    vis = torch.zeros((B, wl.N, wl.D), dtype=torch.int16, device=DEV)
    p = torch.full((B, wl.N), 1.0 / wl.N, dtype=torch.float32, device=DEV)
    keep = torch.empty((B, wl.K), dtype=torch.int32, device=DEV)
    with pytest.raises(mb.MapError) as e:
        ctx.select_noalloc(p, vis, wl.K, keep)
    assert e.value.code == mb.MAP_EUNSUPPORTED
    with pytest.raises(mb.MapError) as e:    # diversity term on: k <= 768, as for map_select
        ctx.select_noalloc(p[:1], vis[:1], 800, torch.empty((1, 800), dtype=torch.int32, device=DEV))
    assert e.value.code == mb.MAP_EUNSUPPORTED
    ctx.close()
