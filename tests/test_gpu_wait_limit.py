"""A bounded device-side wait that runs out, on a tensor-core GEMM: with the wait limit set
to 1 ns the kernel gives up (it stops issuing, lets the copies and MMAs in flight land,
releases its tensor memory and exits), map_status reports MAP_ETIMEOUT once, and the next
call with the default limit computes the right result.  No fault and no hang: every wait
is bounded, and the kernel is a one-SM tile (no peer CTA).  Marked gpu."""
import pytest
import torch

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_06411_gb300 import binding as mb  # noqa: E402
from paper_2608_06411_gb300 import workloads as W  # noqa: E402

DEV = torch.device("cuda:0")


def test_gemm_wait_that_runs_out_reports_timeout_and_the_context_stays_usable():
    dims = W.PredictorDims(D=256, Dh=256, dp=64)
    w = {k: torch.from_numpy(v.view("int16")).to(DEV) for k, v in W.make_weights(dims).items()}
    ctx = mb.Context(w, dims.D, dims.Dh, dims.dp)
    g = torch.Generator(device="cpu").manual_seed(5)
    # one 128 x 256 output tile with K = 16384: the epilogue waits tens of microseconds for it
    x = torch.randn(128, 16384, generator=g).to(torch.bfloat16).to(DEV)
    wt = (torch.randn(256, 16384, generator=g) / 128.0).to(torch.bfloat16).to(DEV)
    b = torch.randn(256, generator=g).to(torch.bfloat16).to(DEV)
    ctx.set_wait_limit(1)
    ctx.linear(x, wt, b, mb.EPI_GELU_BF16)
    assert ctx.status() == mb.MAP_ETIMEOUT
    assert ctx.status() == mb.MAP_OK               # reported once, then cleared
    ctx.set_wait_limit(0)
    y = ctx.linear(x, wt, b, mb.EPI_GELU_BF16)
    torch.cuda.synchronize()
    ctx.check()
    ref = torch.nn.functional.gelu(x.float() @ wt.float().T + b.float())
    torch.testing.assert_close(y.float(), ref, rtol=2 ** -7, atol=2e-3)
    ctx.close()
