"""The roofline arithmetic that bench.py reports: algorithmic FLOPs and bytes per image,
checked against hand-worked counts (CPU only).

Per image, with input width D, MLP width Dh, head width dp, N visual tokens, M question
tokens and k kept tokens, the method needs: both MLPs and projections for every token
(2(D·Dh + Dh·Dh + Dh·dp) per token as written, 2(D·Dh + Dh·dp) with the second layer and the
projection folded into one matrix), the Eq. 3 logits (2·M·N·dp) and the diversity term of
Eq. 4 (2·k·N·D: each retained basis vector against each candidate).  Bytes: the features and
questions once, the scores, the kept tokens read and written, the weights once."""
import sys
from pathlib import Path

import numpy as np
import pytest

sys.path.insert(0, str(Path(__file__).resolve().parents[1]))
import bench  # noqa: E402
from paper_2608_06411_gb300 import workloads as W  # noqa: E402


def test_single_llava_next_image_exact_counts():
    # N = 2880, D = 4096, Dh = 1024, dp = 128, M = 64, k = 160, worked out by hand:
    #   per token as written: 2 (4096*1024 + 1024*1024 + 1024*128) = 10 747 904
    #   folded:               2 (4096*1024 + 1024*128)             =  8 650 752
    #   visual 2880 tokens, text 64 tokens, logits 2*64*2880*128 = 47 185 920,
    #   diversity 2*160*2880*4096 = 3 774 873 600
    dims = W.PredictorDims()
    lens = np.array([64])
    as_written = 2880 * 10_747_904 + 64 * 10_747_904 + 47_185_920 + 3_774_873_600
    folded = 2880 * 8_650_752 + 64 * 8_650_752 + 47_185_920 + 3_774_873_600
    assert as_written == 35_463_888_896 and folded == 29_289_873_408
    assert bench.method_as_written_flops(dims, 2880, 160, lens) == as_written
    flops, bytes_ = bench.algorithmic(dims, 2880, 160, lens)
    assert flops == folded
    # bytes: V 2880*4096*2, T 64*4096*2, scores 2880*4, kept tokens read + written 2*160*4096*2,
    # folded weights (4096*1024 + 1024*128) * 2 matrices * 2 bytes
    assert bytes_ == 23_592_960 + 524_288 + 11_520 + 2_621_440 + 17_301_504


@pytest.mark.parametrize("key,gflop_per_image", [("c0", 6.69), ("c1", 35.5), ("c3", 36.3), ("c4", 95.0)])
def test_per_image_counts_of_the_configurations(key, gflop_per_image):
    # hand-tabulated per-image GFLOP as the method is written (question lengths at their
    # stated means for the batched configurations, hence the 1% tolerance)
    wl = W.WORKLOADS[key]
    dims = W.PredictorDims(D=wl.D)
    lens = W.make_lens(wl)
    got = bench.method_as_written_flops(dims, wl.N, wl.K, lens) / len(lens) / 1e9
    assert got == pytest.approx(gflop_per_image, rel=1e-2)


def test_batched_step_roofline_time():
    # 64 LLaVA-NeXT images at the measured 1953.3 TFLOP/s bf16 peak: about 1.19 ms as written
    # (the batch is tensor-bound: its 1.77 GB take 0.27 ms at 6675.5 GB/s)
    wl = W.WORKLOADS["c3"]
    dims = W.PredictorDims()
    lens = W.make_lens(wl)
    t_flop = bench.method_as_written_flops(dims, wl.N, wl.K, lens) / 1953.3e12
    _, bytes_ = bench.algorithmic(dims, wl.N, wl.K, lens)
    assert t_flop == pytest.approx(1.19e-3, rel=1e-2)
    assert bytes_ / 6675.5e9 < 0.3 * t_flop
