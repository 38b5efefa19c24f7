"""Benchmark of the MAP pruning path (score -> select -> gather) on GB300.

Workload: batched serving shaped like LLaVA-NeXT-7B (64 images per GPU, N = 2880 visual
tokens of width 4096 each, question lengths uniform in [16, 256], keep k = 160 per image,
10% near-duplicate images), seeded synthetic inputs (the paper's benchmark images and
questions are not available).  One step = map_prune over the whole batch with the inputs
already in HBM.  Prints one JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

--impl reference times the CPU oracle on the host cores instead (a bounded sample of the
same workload per step).  Under torchrun each rank runs 64 images of its own (weak
scaling); there is no collective on the data path.
"""
from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import math
import os
import subprocess
import sys
import threading
import time

# The CPU oracle's BLAS uses every host core; set before numpy is imported.
_CORES = os.cpu_count() or 1
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(_CORES))

import numpy as np  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_06411_gb300 import workloads as W  # noqa: E402
from paper_2608_06411_gb300.sharding import image_range, max_over_ranks  # noqa: E402

METRIC = "images pruned/s (score+select+gather) at N=2880,k=160; p50/p99 µs; % roofline"
WORKLOAD = W.WORKLOADS["c3"]
DATA = "synthetic (seeded clustered features and N(0,1) questions, LLaVA-NeXT-7B shapes)"
DIMS = W.PredictorDims()


def algorithmic(dims, N, K, lens):
    """Algorithmic FLOPs and HBM bytes of one batch (what the method needs):
    predictor GEMMs for every visual and question token (layer 1, then the second layer and
    the W_K / W_Q projection as one folded Dh x dp matrix, since nothing lies between them),
    the Eq. 3 logits, and 2*K*N*D for the diversity term (each retained basis vector against
    each candidate); bytes = the features read once, scores written, kept tokens read and
    written, weights read once."""
    D, Dh, dp = dims.D, dims.Dh, dims.dp
    per_tok = 2 * (D * Dh + Dh * dp)
    B = len(lens)
    M = int(np.sum(lens))
    flops = B * N * per_tok + M * per_tok + 2 * M * N * dp + B * 2 * K * N * D
    weights = 2 * (D * Dh + Dh * dp) * 2
    bytes_ = B * N * D * 2 + M * D * 2 + B * N * 4 + 2 * B * K * D * 2 + weights
    return flops, bytes_


def method_as_written_flops(dims, N, K, lens):
    """The same count with the second MLP layer and the projection as separate matrices
    (2 Dh^2 + 2 Dh dp per token instead of 2 Dh dp), as the method is written."""
    D, Dh, dp = dims.D, dims.Dh, dims.dp
    per_tok = 2 * (D * Dh + Dh * Dh + Dh * dp)
    B = len(lens)
    M = int(np.sum(lens))
    return B * N * per_tok + M * per_tok + 2 * M * N * dp + B * 2 * K * N * D


def bench_qcts(mb, dev, stream, steps, hbm, cpu_on, samples=None):
    """Question Contrastive Teacher Selection (Eq. 1-2) on LLaVA-NeXT-7B-shaped attention
    maps: 2 samples x 32 layers x 32 heads, N = 2880, questions U[16,128] tokens and a
    7-token reference question (1.1 GB of bf16 maps, larger than L2).  Timed with CUDA
    events around each map_qcts call (all three of its launches)."""
    import torch
    wq = W.ATTENTION_WORKLOADS["q1"]
    if samples is not None and samples != wq.B:
        wq = dataclasses.replace(wq, B=samples)
    attn_np, lens, ref_np = W.make_attention_batch(wq, threads=min(16, _CORES))
    attn = torch.from_numpy(attn_np.view(np.int16)).to(dev)
    ref = torch.from_numpy(ref_np.view(np.int16)).to(dev)
    B, L, N = wq.B, wq.L, wq.N
    outs = [torch.empty((B, L, N), dtype=torch.float32, device=dev) for _ in range(2)]
    js = torch.empty((B, L), dtype=torch.float32, device=dev)
    teacher = torch.empty(B, dtype=torch.int32, device=dev)
    tp = torch.empty((B, N), dtype=torch.float32, device=dev)

    def call():
        mb.qcts(attn, lens, ref, L, wq.H, N, outs[0], outs[1], js, teacher, tp)

    for _ in range(3):
        call()
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    evs[0].record(stream)
    for i in range(steps):
        call()
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    ms = np.array([evs[i].elapsed_time(evs[i + 1]) for i in range(steps)])
    avg_s = evs[0].elapsed_time(evs[-1]) / 1000.0 / steps
    bytes_ = attn_np.nbytes + ref_np.nbytes + 2 * B * L * N * 4 + B * L * 4 + B * 4 + B * N * 4
    res = {"workload": wq.name, "samples": B, "L": L, "H": wq.H, "N": N,
           "question_len": [int(x) for x in lens], "ref_len": wq.m_ref,
           "value": B / avg_s, "unit": "samples/s", "us_per_call_p50": float(np.percentile(ms, 50) * 1000),
           "us_per_call_p99": float(np.percentile(ms, 99) * 1000),
           "roofline": {"bound": "hbm", "kernel": "map_qcts (column sums, normalise + JS, teacher)",
                        "achieved": bytes_ / avg_s / 1e9, "peak": hbm, "unit": "GB/s",
                        "frac": bytes_ / avg_s / 1e9 / hbm, "algorithmic_bytes": int(bytes_)}}
    if cpu_on:
        from oracle import qcts_oracle as Q
        one = attn_np[:L * wq.H * int(lens[0]) * N]
        t0 = time.perf_counter()
        Q.qcts_batch(one, lens[:1], ref_np[:1], L, wq.H, N)
        secs = time.perf_counter() - t0
        res["cpu_baseline"] = {"value": 1.0 / secs, "unit": "samples/s", "cores": _CORES, "kind": "oracle",
                               "sample": f"sample 0 of the batch ({int(lens[0])} question tokens), numpy float64, "
                                         f"{secs:.1f} s"}
    del attn, ref
    return res


def bench_ragged(mb, dev, stream, steps, bf16_peak, hbm):
    """Ragged batch (Qwen2.5-VL-style variable resolution): 16 images of 675-1222 tokens in
    a batch padded to 1280, D = 3584, keep 128, through map_prune_ragged on device buffers."""
    import torch
    wr = W.RAGGED_WORKLOADS["c5"]
    vis_np, text_np, lens, nv = W.make_ragged_batch(wr, threads=min(16, _CORES))
    dims = W.PredictorDims(D=wr.D)
    w = W.make_weights(dims)
    ctx = mb.Context({k: torch.from_numpy(v.view(np.int16)).to(dev) for k, v in w.items()}, dims.D, dims.Dh,
                     dims.dp)
    vis = torch.from_numpy(vis_np.view(np.int16)).to(dev)
    text = torch.from_numpy(text_np.view(np.int16)).to(dev)
    B, N, K = wr.B, wr.n_max, wr.K
    out = torch.empty((B, K, wr.D), dtype=torch.int16, device=dev)
    keep = torch.empty((B, K), dtype=torch.int32, device=dev)
    sc = torch.empty((B, N), dtype=torch.float32, device=dev)
    for _ in range(3):
        ctx.prune_ragged(text, vis, lens, nv, K, out, keep, sc)
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    evs[0].record(stream)
    for i in range(steps):
        ctx.prune_ragged(text, vis, lens, nv, K, out, keep, sc)
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    ctx.check()
    ctx.close()
    ms = np.array([evs[i].elapsed_time(evs[i + 1]) for i in range(steps)])
    step_s = evs[0].elapsed_time(evs[-1]) / 1000.0 / steps
    # algorithmic work of the valid tokens only (the padding rows are the layout's overhead)
    flops = sum(algorithmic(dims, int(nv[b]), K, lens[b:b + 1])[0] for b in range(B))
    bytes_ = sum(algorithmic(dims, int(nv[b]), K, lens[b:b + 1])[1] for b in range(B))
    t_roof = max(flops / (bf16_peak * 1e12), bytes_ / (hbm * 1e9))
    return {"workload": wr.name, "B": B, "n_max": N, "n_valid": [int(x) for x in nv], "D": wr.D, "k": K,
            "value": B / step_s, "unit": "images/s", "ms_per_batch_p50": float(np.percentile(ms, 50)),
            "ms_per_batch_p99": float(np.percentile(ms, 99)),
            "step_roofline": {"algorithmic_gflop_per_image": flops / B / 1e9, "t_roofline_ms": t_roof * 1000,
                              "frac": t_roof / step_s, "bound": "tensor", "peak_source": "measured bf16 burst"}}


def distill_tensor_flops(dims, N, lens):
    """FLOPs the distillation step's contractions perform on the tensor cores: each runs as
    one bf16 GEMM over K' = n ceil64(K) (n = 1 for two bf16 operands, 3 for an fp32 against a
    bf16 one, 6 for two fp32 operands: the split-bf16 terms down to 2^-24), and the
    algorithmic (fp32) FLOPs 2 M N K of the same list."""
    D, Dh, dp = dims.D, dims.Dh, dims.dp
    B = len(lens)
    Tv, Tt = B * N, int(np.sum(lens))
    mms = []
    for T in (Tv, Tt):
        mms += [(T, Dh, D, 1), (T, Dh, Dh, 3), (T, dp, Dh, 3)]                        # forward
        mms += [(dp, Dh, T, 6), (T, Dh, dp, 3), (Dh, Dh, T, 6), (T, Dh, Dh, 3), (Dh, D, T, 3)]   # backward
    for m in lens:
        m = int(m)
        mms += [(m, N, dp, 6), (m, dp, N, 6), (N, dp, m, 6)]                          # logits, dq, dk
    performed = sum(2 * M * Nn * n * ((K + 63) // 64 * 64) for M, Nn, K, n in mms)
    algorithmic = sum(2 * M * Nn * K for M, Nn, K, n in mms)
    return performed, algorithmic


def bench_distill(mb, dev, stream, steps, cpu_on, bf16_peak=None):
    """Predictor distillation step (KL loss + gradients of every weight) on 4 LLaVA-NeXT-shaped
    training samples: N = 2880 visual tokens, questions U[16,128], D = 4096, Dh = 1024,
    dp = 128.  The contractions run on the tcgen05 GEMM with split-bf16 operands (fp32-level
    products), so the roofline is the bf16 tensor peak against the tensor work performed."""
    import torch
    wl = W.WORKLOADS["c1"]
    B, N = 4, wl.N
    dims = W.PredictorDims()
    rng = np.random.Generator(np.random.PCG64(4242))
    lens = rng.integers(16, 129, size=B).astype(np.int32)
    vis_np = np.stack([W.make_image(wl, 100 + b) for b in range(B)])
    text_np = np.concatenate([W.make_text(wl, 100 + b, int(lens[b])) for b in range(B)])
    t = rng.gamma(0.3, size=(B, N))
    teacher_np = (t / t.sum(axis=1, keepdims=True)).astype(np.float32)
    w = W.make_weights(dims, bias_std=0.1)
    ctx = mb.Context({k: torch.from_numpy(v.view(np.int16)).to(dev) for k, v in w.items()}, dims.D, dims.Dh,
                     dims.dp)
    vis = torch.from_numpy(vis_np.view(np.int16)).to(dev)
    text = torch.from_numpy(text_np.view(np.int16)).to(dev)
    teacher = torch.from_numpy(teacher_np).to(dev)
    loss, grads = ctx.distill_grad(text, vis, lens, teacher)
    for _ in range(2):
        ctx.distill_grad(text, vis, lens, teacher, grads, loss)
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    evs[0].record(stream)
    for i in range(steps):
        ctx.distill_grad(text, vis, lens, teacher, grads, loss)
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    ctx.check()
    ctx.close()
    step_s = evs[0].elapsed_time(evs[-1]) / 1000.0 / steps
    performed, algorithmic = distill_tensor_flops(dims, N, lens)
    peak = bf16_peak if bf16_peak else measured_peaks()[1]
    achieved = performed / step_s / 1e12
    res = {"workload": "distill_llava_next_b4_n2880", "B": B, "N": N, "question_len": [int(x) for x in lens],
           "value": B / step_s, "unit": "samples/s", "ms_per_step": step_s * 1000,
           "roofline": {"bound": "tensor", "kernel": "whole step: split-bf16 tcgen05 GEMMs, operand staging, "
                                                     "elementwise and reduction kernels",
                        "achieved": achieved, "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                        "tensor_gflop_performed": performed / 1e9, "algorithmic_gflop": algorithmic / 1e9,
                        "fp32_equivalent_tflops": algorithmic / step_s / 1e12,
                        "peak_source": "measured bf16 burst"}}
    if cpu_on:
        from oracle import distill_oracle as DO
        t0 = time.perf_counter()
        DO.distill_batch(text_np[:int(lens[0])], vis_np[:1], lens[:1], teacher_np[:1].astype(np.float64), w)
        secs = time.perf_counter() - t0
        res["cpu_baseline"] = {"value": 1.0 / secs, "unit": "samples/s", "cores": _CORES, "kind": "oracle",
                               "sample": f"sample 0 ({int(lens[0])} question tokens), numpy float64, {secs:.1f} s"}
    return res


def bench_config(mb, dev, stream, key, steps, bf16_peak, hbm, ctx=None):
    """One more workload of the pruning path through map_prune on device buffers: per-batch
    CUDA-event times (p50/p99) and the fraction of the algorithmic roofline (GEMM FLOPs at
    the measured bf16 peak vs feature bytes at the measured HBM rate; FLOPs counted as the
    method is written and, stricter, with the folded second layer)."""
    import torch
    wl = W.WORKLOADS[key]
    dims = W.PredictorDims(D=wl.D)
    vis_np, text_np, lens = W.make_batch(wl, threads=min(16, _CORES))
    own = ctx is None
    if own:
        w = W.make_weights(dims)
        ctx = mb.Context({k: torch.from_numpy(v.view(np.int16)).to(dev) for k, v in w.items()}, dims.D, dims.Dh,
                         dims.dp)
    vis = torch.from_numpy(vis_np.view(np.int16)).to(dev)
    text = torch.from_numpy(text_np.view(np.int16)).to(dev)
    B, N, K = wl.B, wl.N, wl.K
    out = torch.empty((B, K, wl.D), dtype=torch.int16, device=dev)
    keep = torch.empty((B, K), dtype=torch.int32, device=dev)
    sc = torch.empty((B, N), dtype=torch.float32, device=dev)
    for _ in range(5):
        ctx.prune(text, vis, lens, K, out, keep, sc)
    torch.cuda.synchronize()
    ms = []
    for i in range(steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ctx.prune(text, vis, lens, K, out, keep, sc)
        e1.record(stream)
        torch.cuda.synchronize()
        ms.append(e0.elapsed_time(e1))
    ctx.check()
    if own:
        ctx.close()
    ms = np.array(ms)
    t = float(np.median(ms)) / 1000.0
    flops, bytes_ = algorithmic(dims, N, K, lens)
    flops_w = method_as_written_flops(dims, N, K, lens)
    t_fold = max(flops / (bf16_peak * 1e12), bytes_ / (hbm * 1e9))
    t_writ = max(flops_w / (bf16_peak * 1e12), bytes_ / (hbm * 1e9))
    return {"workload": wl.name, "B": B, "N": N, "D": wl.D, "k": K,
            "question_len": f"U[{wl.m_lo},{wl.m_hi}], sum={int(np.sum(lens))}" if B > 1 else int(lens[0]),
            "value": B / t, "unit": "images/s", "us_per_batch_p50": float(np.percentile(ms, 50) * 1000),
            "us_per_batch_p99": float(np.percentile(ms, 99) * 1000), "batches_timed": steps,
            "step_roofline": {"algorithmic_gflop_per_image": flops_w / B / 1e9, "t_roofline_us": t_writ * 1e6,
                              "frac": t_writ / t, "frac_folded": t_fold / t,
                              "bound": "tensor" if flops_w / (bf16_peak * 1e12) > bytes_ / (hbm * 1e9) else "hbm",
                              "peak_source": "measured bf16 burst, hbm"}}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d["bf16_tflops_sustained"], "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def profile_traffic(kernel_file: str):
    """DRAM bytes per launch of the f_V layer-1 GEMM from the committed ncu summary, if
    the kernel source has not changed since it was captured."""
    src = os.path.join(ROOT, "paper_2608_06411_gb300", "csrc", "gemm_tc.cu")
    path = os.path.join(ROOT, "profiles", kernel_file)
    if not os.path.exists(path):
        return None
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    info = {}
    for line in open(path):
        if ":" in line:
            k, v = line.split(":", 1)
            info[k.strip()] = v.strip()
    if info.get("source_sha256_16") != h:
        return None
    try:
        return float(info["dram_bytes_per_launch_full"])
    except (KeyError, ValueError):
        return None


class ClockSampler:
    """SM clock and clock-event reasons while the timed region runs.  NVML through ctypes,
    polled every 5 ms (reading only), when libnvidia-ml loads; else nvidia-smi -lms 50.
    mark()/stop() bracket the timed region; only samples taken inside it are reported."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASON_BITS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown"}

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.nvml = None
        self.samples = []          # (time, sm_mhz, sm_max_mhz, reasons)
        self.t0 = None
        self.stop_flag = False

    def _nvml_handle(self):
        import ctypes
        lib = ctypes.CDLL("libnvidia-ml.so.1")
        if lib.nvmlInit_v2() != 0:
            return None
        h = ctypes.c_void_p()
        vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")
        entry = vis[self.gpu].strip() if vis and vis[0] != "" and self.gpu < len(vis) else str(self.gpu)
        if entry.isdigit():
            rc = lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(int(entry)), ctypes.byref(h))
        else:
            rc = lib.nvmlDeviceGetHandleByUUID(entry.encode(), ctypes.byref(h))
        return (lib, h) if rc == 0 else None

    def start(self):
        try:
            self.nvml = self._nvml_handle()
        except OSError:
            self.nvml = None
        if self.nvml:
            self.t = threading.Thread(target=self._poll_nvml, daemon=True)
            self.t.start()
            return
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "50"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read_smi, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _poll_nvml(self):
        import ctypes
        lib, h = self.nvml
        clk, cmax, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        get_reasons = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            lib.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self.stop_flag:
            ok = lib.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0      # NVML_CLOCK_SM
            lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(cmax))
            get_reasons(h, ctypes.byref(rs))
            if ok:
                names = [n for bit, n in self.REASON_BITS.items() if rs.value & bit]
                self.samples.append((time.perf_counter(), float(clk.value), float(cmax.value), names))
            time.sleep(0.005)

    def _read_smi(self):
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.strip().split(",")]
            if len(parts) < 9:
                continue
            try:
                sm, smax = float(parts[1]), float(parts[2])
            except ValueError:
                continue
            rs = [nm for nm, v in zip(names, parts[5:9]) if v.lower().startswith("active")]
            self.samples.append((time.perf_counter(), sm, smax, rs))

    def mark(self):
        self.t0 = time.perf_counter()

    def stop(self):
        t1 = time.perf_counter()
        if not self.nvml and not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["clock sampling unavailable"], "samples": 0}
        self.stop_flag = True
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.t.join(timeout=5)
        inside = [x for x in self.samples if self.t0 is None or self.t0 <= x[0] <= t1]
        if not inside and self.samples:           # region shorter than one sample period
            inside = [min(self.samples, key=lambda x: abs(x[0] - t1))]
        sm = [x[1] for x in inside]
        reasons = sorted({r for x in inside for r in x[3]})
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": inside[-1][2] if inside else None,
                "reasons": reasons, "samples": len(sm), "source": "nvml" if self.nvml else "nvidia-smi"}


def time_oracle(n_images: int, first_image: int = 0) -> float:
    """Seconds the oracle spends on n_images (input generation excluded)."""
    from oracle import map_oracle as O
    w = W.make_weights(DIMS)
    lens_all = W.make_lens(WORKLOAD)
    total = 0.0
    for i in range(first_image, first_image + n_images):
        vis = W.make_image(WORKLOAD, i)
        text = W.make_text(WORKLOAD, i, int(lens_all[i % len(lens_all)]))
        t0 = time.perf_counter()
        p = O.map_score(text, vis[None], [len(text)], w)[0]
        r = O.select(p, O.bf16_bits_to_f64(vis), WORKLOAD.K, O.resolve_k0(WORKLOAD.K))
        O.gather(vis[None], r["keep"][None])
        total += time.perf_counter() - t0
    return total


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


REF_BUDGET_S = 150.0


def workload_config(lens, ws):
    """The benchmarked workload: the batched-serving configuration (LLaVA-NeXT-7B shapes)."""
    return {"workload": WORKLOAD.name, "B": WORKLOAD.B, "N": WORKLOAD.N, "D": WORKLOAD.D, "k": WORKLOAD.K,
            "Dh": DIMS.Dh, "dp": DIMS.dp,
            "question_len": f"U[{WORKLOAD.m_lo},{WORKLOAD.m_hi}], sum={int(np.sum(lens))}",
            "k0": "k/2", "lambda": 1.0, "near_duplicate_images": "b % 10 == 0",
            "l2": "inputs larger than L2 (1.51 GB of features per step)",
            "parallelism": f"replicas x{ws}, 64 images per GPU"}


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    for _ in range(args.warmup):
        pass                                   # the oracle has no warm-up state
    per_step = []
    t0 = time.perf_counter()
    for s in range(args.steps):              # bounded: stop once REF_BUDGET_S of oracle time is spent
        per_step.append(time_oracle(1, first_image=s % WORKLOAD.B))
        if time.perf_counter() - t0 > REF_BUDGET_S:
            break
    total = float(np.sum(per_step))
    value = len(per_step) / total
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": args.gpus,
        "steps": args.steps, "steps_timed": len(per_step), "warmup": args.warmup,
        "ms_per_step": 1000 * total / len(per_step),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": DATA,
        "config": workload_config(W.make_lens(WORKLOAD), ws),
        "cpu_baseline": {"value": value, "unit": "images/s", "cores": _CORES, "kind": "oracle",
                         "sample": f"{len(per_step)} images of the 64-image batch, one per step (at most "
                                   f"{REF_BUDGET_S:.0f} s of oracle time), numpy float64 oracle"},
        "e2e": {"value": value, "unit": "images/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-images", type=int, default=1, help="oracle images timed for cpu_baseline")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--no-qcts", action="store_true", help="skip the teacher-selection (QCTS) measurement")
    ap.add_argument("--only-qcts", action="store_true",
                    help="run only the teacher-selection measurement (for profiling), print its JSON")
    ap.add_argument("--qcts-samples", type=int, default=W.ATTENTION_WORKLOADS["q1"].B)
    ap.add_argument("--only-config", choices=["c0", "c4"], default=None,
                    help="time only that configuration through map_prune (for profiling), print its JSON")
    ap.add_argument("--only-distill", action="store_true",
                    help="run only the distillation-step measurement (for profiling), print its JSON")
    ap.add_argument("--batch", type=int, default=WORKLOAD.B, help="images per GPU (profiling on a smaller case)")
    ap.add_argument("--minimal", action="store_true",
                    help="time the steps only (no clock sampling, latency, e2e or CPU baseline): for ncu runs")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    args.warmup = max(3, args.warmup)

    import torch
    from paper_2608_06411_gb300 import binding as mb

    ws, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if args.only_config:
        if rank == 0:
            hbm, bf16_burst, _, _ = measured_peaks()
            print(json.dumps(bench_config(mb, dev, torch.cuda.current_stream(), args.only_config, args.steps,
                                          bf16_burst, hbm)))
        return 0
    if args.only_distill:
        if rank == 0:
            print(json.dumps(bench_distill(mb, dev, torch.cuda.current_stream(), args.steps, False)))
        return 0
    if args.only_qcts:
        if rank == 0:
            hbm = measured_peaks()[0]
            print(json.dumps(bench_qcts(mb, dev, torch.cuda.current_stream(), args.steps, hbm, False,
                                        args.qcts_samples)))
        return 0
    pg = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist

    B, N, K, D = args.batch, WORKLOAD.N, WORKLOAD.K, WORKLOAD.D
    first, B = image_range(B * ws, ws, rank)              # weak scaling: 64 images per rank
    vis_np, text_np, lens = W.make_batch(WORKLOAD, B=B, first_image=first, threads=min(16, _CORES))
    w = W.make_weights(DIMS)
    ctx = mb.Context({k: torch.from_numpy(v.view(np.int16)).to(dev) for k, v in w.items()}, DIMS.D, DIMS.Dh,
                     DIMS.dp)
    vis = torch.from_numpy(vis_np.view(np.int16)).to(dev)
    text = torch.from_numpy(text_np.view(np.int16)).to(dev)
    out = torch.empty((B, K, D), dtype=torch.int16, device=dev)
    keep = torch.empty((B, K), dtype=torch.int32, device=dev)
    scores = torch.empty((B, N), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        ctx.prune(text, vis, lens, K, out, keep, scores)

    sampler = ClockSampler(local)          # started early: nvidia-smi start-up stalls the device briefly
    if not args.minimal:
        sampler.start()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    ctx.check()
    if not args.minimal:
        time.sleep(1.0)
        for _ in range(2):
            step()
        torch.cuda.synchronize()

    # ---------------------------------------------------------------- timed region
    ctx.set_timing(True)
    for kid in range(7):
        ctx.read_timing(kid)                    # reset
    launches0 = ctx.counters()["launches"]
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    sampler.mark()
    evs[0].record(stream)
    for i in range(args.steps):
        step()
        evs[i + 1].record(stream)
    torch.cuda.synchronize()
    if pg:
        pg.barrier()
    clocks = sampler.stop()
    launches = ctx.counters()["launches"] - launches0
    ctx.check()
    step_ms = np.array([evs[i].elapsed_time(evs[i + 1]) for i in range(args.steps)])
    total_ms = evs[0].elapsed_time(evs[-1])
    fv1_ms, fv1_n = ctx.read_timing(mb.K_GEMM_FV1)
    other = {name: ctx.read_timing(kid) for name, kid in
             [("wk", mb.K_GEMM_WK), ("text_stream_span", mb.K_GEMM_TEXT), ("scores", mb.K_SCORES),
              ("select", mb.K_SELECT), ("gather", mb.K_GATHER)]}
    ctx.set_timing(False)
    total_ms = max_over_ranks(total_ms, dev)

    images = B * args.steps * ws
    value = images / (total_ms / 1000.0)
    hbm, bf16_burst, bf16_sust, peak_src = measured_peaks()
    sustained = total_ms > 2000.0
    peak = bf16_sust if sustained else bf16_burst
    fv1_flops = 2.0 * B * N * DIMS.D * DIMS.Dh
    fv1_avg_s = fv1_ms / 1000.0 / max(1, fv1_n)
    achieved = fv1_flops / fv1_avg_s / 1e12
    traffic = profile_traffic("gemm_fv1_c3.txt")
    flops, bytes_ = algorithmic(DIMS, N, K, lens)
    t_roof = max(flops / (bf16_burst * 1e12), bytes_ / (hbm * 1e9))
    step_s = total_ms / 1000.0 / args.steps

    if args.minimal:
        if rank == 0:
            print(json.dumps({"metric": METRIC, "value": B * args.steps * ws / (total_ms / 1000.0), "unit": "images/s",
                              "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
                              "ms_per_step": total_ms / args.steps, "higher_is_better": True, "scaling": "weak",
                              "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                              "config": {"workload": WORKLOAD.name, "B": B, "minimal": True},
                              "gpu_launches": int(launches)}))
        ctx.close()
        if pg:
            pg.destroy_process_group()
        return 0

    # ---------------------------------------------------------------- single-image latency (N=2880, k=160)
    w1 = W.WORKLOADS["c1"]
    v1 = torch.from_numpy(W.make_image(w1, 0).view(np.int16)).to(dev)[None].contiguous()
    t1 = torch.from_numpy(W.make_text(w1, 0, 64).view(np.int16)).to(dev)
    o1 = torch.empty((1, w1.K, D), dtype=torch.int16, device=dev)
    k1 = torch.empty((1, w1.K), dtype=torch.int32, device=dev)
    s1 = torch.empty((1, w1.N), dtype=torch.float32, device=dev)
    lat = []
    for i in range(1010):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        ctx.prune(t1, v1, [64], w1.K, o1, k1, s1)
        e1.record(stream)
        torch.cuda.synchronize()
        if i >= 10:
            lat.append(e0.elapsed_time(e1) * 1000.0)

    # ---------------------------------------------------------------- end to end from host buffers
    vis_h = torch.from_numpy(vis_np.view(np.int16)).pin_memory()
    text_h = torch.from_numpy(text_np.view(np.int16)).pin_memory()
    out_h = torch.empty((B, K, D), dtype=torch.int16).pin_memory()
    keep_h = torch.empty((B, K), dtype=torch.int32).pin_memory()
    for _ in range(3):                                    # warm (first pinned-buffer uses)
        ctx.prune(text_h, vis_h, lens, K, out_h, keep_h)
    if pg:
        pg.barrier()
    t0 = time.perf_counter()
    for _ in range(args.e2e_steps):
        ctx.prune(text_h, vis_h, lens, K, out_h, keep_h)
    e2e_s = time.perf_counter() - t0
    e2e_s = max_over_ranks(e2e_s, dev)
    e2e_value = B * args.e2e_steps * ws / e2e_s
    ctx.check()
    # context for the end-to-end figure: this machine's plain pinned host -> device copy rate
    vis_tmp = torch.empty_like(vis)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(3):
        vis_tmp.copy_(vis_h, non_blocking=True)
    torch.cuda.synchronize()
    h2d_gbs = 3 * vis_np.nbytes / (time.perf_counter() - t0) / 1e9
    del vis_tmp

    # ---------------------------------------------------------------- hand-off sequence (kept + question tokens)
    step()
    torch.cuda.synchronize()
    rows = B * K + int(np.sum(lens))
    seq = torch.empty((rows, D), dtype=torch.int16, device=dev)
    pos = torch.empty(rows, dtype=torch.int32, device=dev)
    for _ in range(3):
        ctx.assemble(vis, keep, text, lens, 0, seq, pos)
    hev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    hev[0].record(stream)
    for _ in range(20):
        ctx.assemble(vis, keep, text, lens, 0, seq, pos)
    hev[1].record(stream)
    torch.cuda.synchronize()
    ctx.check()
    h_s = hev[0].elapsed_time(hev[1]) / 1000.0 / 20
    h_bytes = 2 * rows * D * 2 + rows * 4 + B * K * 4
    handoff = {"us_per_call": h_s * 1e6, "rows": rows,
               "roofline": {"bound": "hbm", "kernel": "assemble_kernel (kept tokens + questions, position ids)",
                            "achieved": h_bytes / h_s / 1e9, "peak": hbm, "unit": "GB/s",
                            "frac": h_bytes / h_s / 1e9 / hbm, "algorithmic_bytes": int(h_bytes)}}
    del seq, pos

    ragged = bench_ragged(mb, dev, stream, 20, bf16_burst, hbm) if rank == 0 else None
    c0 = bench_config(mb, dev, stream, "c0", 200, bf16_burst, hbm, ctx) if rank == 0 else None
    c4 = bench_config(mb, dev, stream, "c4", 20, bf16_burst, hbm) if rank == 0 else None

    distill = bench_distill(mb, dev, stream, 5, ws == 1 and not args.no_cpu, bf16_burst) if rank == 0 else None

    qcts = None
    if rank == 0 and not args.no_qcts:
        qcts = bench_qcts(mb, dev, stream, 20, hbm, ws == 1 and not args.no_cpu, args.qcts_samples)

    cpu = None
    if rank == 0 and ws == 1 and not args.no_cpu:
        secs = time_oracle(args.cpu_images)
        cpu = {"value": args.cpu_images / secs, "unit": "images/s", "cores": _CORES, "kind": "oracle",
               "sample": f"{args.cpu_images} image(s) of the batch (N=2880, k=160), numpy float64 oracle, "
                         f"{secs:.1f} s"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "images/s", "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": DATA,
            "config": workload_config(lens, ws),
            "latency_us": {"batch_p50": float(np.percentile(step_ms, 50) * 1000),
                           "batch_p99": float(np.percentile(step_ms, 99) * 1000),
                           "single_image_p50": float(np.percentile(lat, 50)),
                           "single_image_p99": float(np.percentile(lat, 99))},
            "roofline": {"bound": "tensor", "kernel": "f_V layer-1 GEMM (tcgen05)", "achieved": achieved,
                         "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                         "peak_source": f"{peak_src} bf16 {'sustained' if sustained else 'burst'}",
                         "traffic": traffic},
            "step_roofline": {"algorithmic_gflop_per_image": flops / B / 1e9, "t_roofline_ms": t_roof * 1000,
                              "frac": t_roof / step_s,
                              "frac_method_as_written": max(method_as_written_flops(DIMS, N, K, lens) /
                                                            (bf16_burst * 1e12), bytes_ / (hbm * 1e9)) / step_s,
                              "bound": "tensor" if flops / (bf16_burst * 1e12) >
                              bytes_ / (hbm * 1e9) else "hbm", "peak_source": f"{peak_src} bf16 burst, hbm"},
            "kernel_ms_per_step": {"fv1": fv1_ms / args.steps, **{k: v[0] / args.steps for k, v in other.items()}},
            "clocks": clocks,
            "e2e": {"value": e2e_value, "unit": "images/s",
                    "h2d_bytes_per_step": int(vis_np.nbytes + text_np.nbytes),
                    "d2h_bytes_per_step": int(B * K * D * 2 + B * K * 4),
                    "host_to_device_gbs": round(h2d_gbs, 1)},
            "gpu_launches": int(launches),
            "cpu_baseline": cpu,
            "handoff": handoff,
            "ragged": ragged,
            "single_image_c0": c0,
            "high_token_c4": c4,
            "distill": distill,
            "qcts": qcts,
        }
        print(json.dumps(line))
    ctx.close()
    if pg:
        pg.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
