"""map_select_noalloc through the C ABI: same picks as map_select, on two calls in a row.

The allocation-free entry point serves callers that cannot allocate device memory while
they prune (CUDA-graph capture, fixed memory budgets, foreign memory pools); it carves its
workspace from a static device array instead.  This file is collected last on purpose."""
import numpy as np
import pytest
import torch

from paper_2608_06411_gb300 import workloads as W

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_06411_gb300 import binding as mb  # noqa: E402

DEV = torch.device("cuda:0")


def _dev(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def _ctx(D):
    dims = W.PredictorDims(D=D, Dh=256, dp=64)
    w = W.make_weights(dims)
    return mb.Context({k: _dev(v) for k, v in w.items()}, dims.D, dims.Dh, dims.dp)


@pytest.mark.parametrize("wl_name,B,K", [("c0", 1, 32), ("c1", 1, 160), ("c3", 2, 60)])
def test_noalloc_select_matches_map_select(wl_name, B, K):
    wl = W.WORKLOADS[wl_name]
    ctx = _ctx(wl.D)
    vis = np.stack([W.make_image(wl, b) for b in range(B)])
    rng = np.random.default_rng(B * 1000 + K)
    p = torch.from_numpy(rng.dirichlet(np.full(wl.N, 0.3), size=B).astype(np.float32)).to(DEV)
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
    ctx.close()
