"""The predictor distillation step on the GPU (map_distill_grad through the C ABI) against
the float64 oracle: loss D_KL(p* || p_hat) and the gradient of every predictor weight
(section "Cross-Modal Attention Distillation")."""
import numpy as np
import pytest
import torch

from oracle import distill_oracle as DO
from oracle import parity as P
from paper_2608_06411_gb300 import workloads as W

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2608_06411_gb300 import binding as mb  # noqa: E402

DEV = torch.device("cuda:0")


def dev_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(DEV)


def _teachers(B, N, seed):
    rng = np.random.default_rng(seed)
    t = rng.gamma(0.3, size=(B, N))
    t[:, ::7] = 0.0                                    # zero-probability tokens (0 log 0 = 0)
    return (t / t.sum(axis=1, keepdims=True)).astype(np.float32)


def _inputs(wl, B, N, D, lens):
    vis = np.stack([W.make_image(wl, b, N=N, D=D) for b in range(B)])
    text = np.concatenate([W.make_text(wl, b, int(lens[b]), D=D) for b in range(B)])
    return vis, text


def _check(dims, wl, B, N, lens, seed, rope_on=True, bias_std=0.1):
    wts = W.make_weights(dims, seed=seed, bias_std=bias_std)
    ctx = mb.Context({k: dev_bits(v) for k, v in wts.items()}, dims.D, dims.Dh, dims.dp, rope_on=rope_on)
    vis, text = _inputs(wl, B, N, dims.D, lens)
    teacher = _teachers(B, N, seed)
    loss, grads = ctx.distill_grad(dev_bits(text), dev_bits(vis), lens, torch.from_numpy(teacher).to(DEV))
    torch.cuda.synchronize()
    ctx.check()
    ref_loss, ref = DO.distill_batch(text, vis, lens, teacher.astype(np.float64), wts, rope_on=rope_on)
    assert float(loss.item()) == pytest.approx(ref_loss, rel=P.DISTILL_LOSS_RTOL)
    scale = 1e-3 * max(float(np.abs(ref[n]).max()) for n in DO.WEIGHT_NAMES)
    for name in DO.WEIGHT_NAMES:
        err = P.distill_grad_err(grads[name].cpu().numpy(), ref[name], scale)
        assert err <= P.DISTILL_GRAD_TOL, f"{name}: {err:.2e}"
    return ctx, vis, text, teacher, loss, grads


def test_distill_matches_oracle_small():
    _check(W.PredictorDims(D=512, Dh=256, dp=64), W.WORKLOADS["c0"], 3, 200, np.array([5, 17, 9], np.int32), 11)


def test_distill_without_rope():
    _check(W.PredictorDims(D=256, Dh=256, dp=64), W.WORKLOADS["c0"], 2, 130, np.array([3, 1], np.int32), 12,
           rope_on=False)


def test_distill_is_deterministic():
    ctx, vis, text, teacher, loss, grads = _check(W.PredictorDims(D=512, Dh=256, dp=64), W.WORKLOADS["c1"], 2, 300,
                                                  np.array([8, 30], np.int32), 13)
    loss2, grads2 = ctx.distill_grad(dev_bits(text), dev_bits(vis), [8, 30], torch.from_numpy(teacher).to(DEV))
    torch.cuda.synchronize()
    assert float(loss2.item()) == float(loss.item())
    for name in DO.WEIGHT_NAMES:
        assert torch.equal(grads2[name], grads[name]), name


def test_distill_llava_next_shape():
    """Full predictor widths (D = 4096, Dh = 1024, dp = 128), two N = 2880 images."""
    _check(W.PredictorDims(), W.WORKLOADS["c1"], 2, 2880, np.array([64, 23], np.int32), 14)
