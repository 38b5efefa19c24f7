"""Seeded synthetic inputs shaped like the paper's LLaVA-NeXT / Qwen2.5-VL workloads.

This module is the ONE place both the CUDA path and the CPU oracle take their inputs
from.  It holds none of the method's arithmetic: it only draws random numbers and
rounds them to bf16 storage.  Everything is numpy (PCG64), so the same seed gives
the same bytes on x86 and Arm.

Shapes follow the paper's workloads (section "Experiments", Tables 2 and 3):
LLaVA-NeXT-7B feeds N = 2880 visual tokens (5 AnyRes crops of a 24x24 grid) of width
D = 4096 to the language model and keeps K = 160 of them (5.56%); LLaVA-1.5 uses one
24x24 grid (N = 576).  The benchmarks' images and questions are not available, so
visual tokens are drawn as spatially clustered features (cluster centroid + noise),
which gives the diversity term of Eq. 4 real redundancy to remove, and question
tokens are standard normal.

Visual features are returned as uint16 bf16 bit patterns [B, N, D]; question tokens
as packed uint16 [sum(lens), D] plus the per-image lengths.
"""
from __future__ import annotations

import dataclasses
from concurrent.futures import ThreadPoolExecutor

import numpy as np

__all__ = [
    "PredictorDims", "Workload", "WORKLOADS", "f32_to_bf16_bits", "bf16_bits_to_f32",
    "make_weights", "make_image", "make_text", "make_batch", "k0_for",
]


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest, ties to even); return uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    b = np.ascontiguousarray(b, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


@dataclasses.dataclass(frozen=True)
class PredictorDims:
    """Predictor widths.  The paper calls the predictor lightweight but gives no
    widths; these are the reading used throughout (2-layer MLPs of width Dh, one
    query/key head of width dp)."""
    D: int = 4096
    Dh: int = 1024
    dp: int = 128


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    config_id: int
    B: int
    crops: int          # AnyRes crops / tiles per image
    grid: int           # tokens per crop side (24 for LLaVA, 27 for the Qwen-like tiles)
    D: int
    centroids: int      # centroids per crop
    block_rows: int     # centroid grid: rows of blocks per crop
    block_cols: int
    noise: float
    m_lo: int           # question length range (inclusive)
    m_hi: int
    K: int
    near_dup_every: int = 0     # images with b % near_dup_every == 0 repeat crop 0
    near_dup_noise: float = 0.05

    @property
    def N(self) -> int:
        return self.crops * self.grid * self.grid


WORKLOADS = {
    # one 24x24 grid, 16 centroids on 6x6-token blocks, M = 32, keep 32
    "c0": Workload("c0_single_n576", 0, 1, 1, 24, 4096, 16, 4, 4, 0.3, 32, 32, 32),
    # LLaVA-NeXT shape: 5 crops x 24x24, 64 centroids per crop on 3x3 blocks, keep 160
    "c1": Workload("c1_llava_next_n2880", 1, 1, 5, 24, 4096, 64, 8, 8, 0.3, 64, 64, 160),
    # retention sweep reuses the c1 generator (K and the diversity weight vary)
    "c2": Workload("c2_sweep_n2880", 2, 1, 5, 24, 4096, 64, 8, 8, 0.3, 64, 64, 160),
    # batched serving: 64 images, ragged questions, 10% near-duplicate crops
    "c3": Workload("c3_batch64_n2880_k160", 3, 64, 5, 24, 4096, 64, 8, 8, 0.3, 16, 256, 160,
                   near_dup_every=10),
    # high-token regime: 10 tiles x 27x27, D = 3584, 128 centroids per tile, keep 405
    "c4": Workload("c4_batch16_n7290_k405", 4, 16, 10, 27, 3584, 128, 16, 8, 0.3, 32, 512, 405),
}


def _image_rng(config_id: int, image: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(1000 * config_id + image))


def make_image(w: Workload, image: int, N: int | None = None, D: int | None = None) -> np.ndarray:
    """Visual tokens of one image as bf16 bits [N, D].

    Token (r, c) of crop t belongs to block (r * block_rows // grid, c * block_cols // grid)
    of that crop; each block has its own N(0, 1)^D centroid; token = centroid +
    N(0, noise^2).  For near-duplicate images, crops 1.. copy crop 0 plus N(0, 0.05^2).
    """
    D = D or w.D
    rng = _image_rng(w.config_id, image)
    per_crop = w.grid * w.grid
    r = np.arange(w.grid)
    cid = (r[:, None] * w.block_rows // w.grid) * w.block_cols + (r[None, :] * w.block_cols // w.grid)
    cid = cid.reshape(-1)
    dup = w.near_dup_every > 0 and image % w.near_dup_every == 0
    crops = []
    for t in range(w.crops):
        if dup and t > 0:
            crop = crops[0] + rng.standard_normal((per_crop, D), dtype=np.float32) * np.float32(w.near_dup_noise)
        else:
            cent = rng.standard_normal((w.centroids, D), dtype=np.float32)
            crop = cent[cid] + rng.standard_normal((per_crop, D), dtype=np.float32) * np.float32(w.noise)
        crops.append(crop)
    x = np.concatenate(crops, axis=0)
    if N is not None:
        x = x[:N]
    return f32_to_bf16_bits(x)


def make_text(w: Workload, image: int, M: int, D: int | None = None) -> np.ndarray:
    """Question tokens of one image as bf16 bits [M, D], N(0, 1)."""
    D = D or w.D
    rng = np.random.Generator(np.random.PCG64(1000 * w.config_id + image + 1_000_000))
    return f32_to_bf16_bits(rng.standard_normal((M, D), dtype=np.float32))


def make_lens(w: Workload, B: int | None = None) -> np.ndarray:
    """Per-image question lengths, uniform in [m_lo, m_hi]."""
    B = B or w.B
    if w.m_lo == w.m_hi:
        return np.full(B, w.m_lo, dtype=np.int32)
    rng = np.random.Generator(np.random.PCG64(1000 * w.config_id + 999_999))
    return rng.integers(w.m_lo, w.m_hi + 1, size=B).astype(np.int32)


def make_batch(w: Workload, B: int | None = None, first_image: int = 0, threads: int = 8):
    """(vis [B, N, D] u16, text [sum(lens), D] u16, lens [B] int32) for images
    first_image .. first_image + B - 1."""
    B = B or w.B
    lens_all = make_lens(w, max(w.B, first_image + B))
    lens = lens_all[first_image:first_image + B].copy()
    vis = np.empty((B, w.N, w.D), dtype=np.uint16)
    texts = [None] * B

    def one(b):
        vis[b] = make_image(w, first_image + b)
        texts[b] = make_text(w, first_image + b, int(lens[b]))

    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        list(ex.map(one, range(B)))
    text = np.concatenate(texts, axis=0) if B else np.zeros((0, w.D), np.uint16)
    return vis, text, lens


def make_weights(dims: PredictorDims, seed: int = 7, bias_std: float = 0.0) -> dict:
    """Seeded random-init predictor weights as bf16 bits, PyTorch Linear layout [out, in].

    MLP layers: He-normal N(0, 2/fan_in); W_Q, W_K: N(0, 1/fan_in); biases N(0, bias_std^2)
    (zero by default).  With these scales the query-key logits have a standard deviation
    of about 2, so the predicted distribution is far from uniform.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    D, Dh, dp = dims.D, dims.Dh, dims.dp

    def lin(o, i, var):
        return f32_to_bf16_bits(rng.standard_normal((o, i), dtype=np.float32) * np.float32(np.sqrt(var)))

    def bias(o):
        return f32_to_bf16_bits(rng.standard_normal(o, dtype=np.float32) * np.float32(bias_std))

    w = {}
    w["wT1"] = lin(Dh, D, 2.0 / D); w["bT1"] = bias(Dh)
    w["wT2"] = lin(Dh, Dh, 2.0 / Dh); w["bT2"] = bias(Dh)
    w["wQ"] = lin(dp, Dh, 1.0 / Dh)
    w["wV1"] = lin(Dh, D, 2.0 / D); w["bV1"] = bias(Dh)
    w["wV2"] = lin(Dh, Dh, 2.0 / Dh); w["bV2"] = bias(Dh)
    w["wK"] = lin(dp, Dh, 1.0 / Dh)
    return w


def k0_for(K: int, k0_frac: float = 0.5, k0_abs: int = -1) -> int:
    """Size of the initial top-K0 set R0: k0_abs if given, else floor(k0_frac * K),
    clamped to [0, K].  The paper does not state K0; K/2 is the default reading."""
    k0 = k0_abs if k0_abs >= 0 else int(np.floor(k0_frac * K))
    return max(0, min(K, k0))


# ----------------------------------------------------------------------------- QCTS inputs

@dataclasses.dataclass(frozen=True)
class AttentionWorkload:
    """Text-to-vision attention maps of a host MLLM, the input of Question Contrastive
    Teacher Selection (section "Question Contrastive Teacher Selection", Eq. 1-2).

    For each image/question pair: the attention A[l, h, m, n] of question token m to visual
    token n at head h of layer l, for the sample's own question (M_b tokens, ragged) and for
    the fixed reference question (m_ref tokens).  The real maps come from a forward pass of
    the MLLM on the paper's training data, which is not available; these are drawn with the
    LLaVA shapes (L = 32 layers, H = 32 heads for the 7B backbones)."""
    name: str
    config_id: int
    B: int          # image/question pairs
    L: int          # language-model layers
    H: int          # attention heads per layer
    crops: int
    grid: int
    m_lo: int       # question length range (inclusive)
    m_hi: int
    m_ref: int      # tokens of the generic reference question (what the image shows)

    @property
    def N(self) -> int:
        return self.crops * self.grid * self.grid


ATTENTION_WORKLOADS = {
    # LLaVA-1.5-7B: one 24x24 grid
    "q0": AttentionWorkload("q0_llava15_n576", 10, 4, 32, 32, 1, 24, 8, 64, 7),
    # LLaVA-NeXT-7B: 5 AnyRes crops of 24x24
    "q1": AttentionWorkload("q1_llava_next_n2880", 11, 2, 32, 32, 5, 24, 16, 128, 7),
}


def attention_lens(w: AttentionWorkload, B: int | None = None) -> np.ndarray:
    """Question lengths M_b, uniform in [m_lo, m_hi]."""
    B = B or w.B
    rng = np.random.Generator(np.random.PCG64(1000 * w.config_id + 999_999))
    return rng.integers(w.m_lo, w.m_hi + 1, size=B).astype(np.int32)


def make_attention(w: AttentionWorkload, sample: int, M: int, ref: bool = False, L: int | None = None,
                   H: int | None = None, N: int | None = None, threads: int = 8) -> np.ndarray:
    """Attention of one sample as bf16 bits [L, H, M, N].

    Structure shared by both questions of a sample: a log-normal visual saliency per token
    (the generic attention an image draws) and one rectangular region of interest in one
    crop.  The sample's own question additionally pulls attention onto that region in the
    middle layers: the pull has a Gaussian profile over layers, peaked at a random layer in
    the middle half, scaled per head.  Every row gets log-normal noise and a random share in
    [0.05, 0.5] of the query's attention mass (the rest goes to non-visual keys), so rows do
    not sum to one.
    """
    L = L or w.L
    H = H or w.H
    N = N or w.N
    base = np.random.Generator(np.random.PCG64(1000 * w.config_id + sample))
    sal = base.standard_normal(N, dtype=np.float32) * np.float32(0.5)
    roi = np.zeros(N, dtype=np.float32)
    g = w.grid
    crop = int(base.integers(w.crops))
    rh, rw = (int(x) for x in base.integers(4, min(g, 10) + 1, size=2))
    r0, c0 = int(base.integers(0, g - rh + 1)), int(base.integers(0, g - rw + 1))
    rr, cc = np.meshgrid(np.arange(r0, r0 + rh), np.arange(c0, c0 + rw), indexing="ij")
    idx = crop * g * g + rr.reshape(-1) * g + cc.reshape(-1)
    roi[idx[idx < N]] = 1.0
    l_peak = int(base.integers(L // 4, 3 * L // 4 + 1))
    layer_gain = 3.0 * np.exp(-0.5 * ((np.arange(L) - l_peak) / max(L / 8.0, 1.0)) ** 2)
    head_gain = base.uniform(0.3, 1.2, H)
    out = np.empty((L, H, M, N), dtype=np.uint16)

    def layer(l):
        rng = np.random.Generator(np.random.PCG64([1000 * w.config_id + sample, int(ref), l]))
        z = rng.standard_normal((H, M, N), dtype=np.float32) * np.float32(0.7)
        z += sal
        if not ref:
            z += (layer_gain[l] * head_gain).astype(np.float32)[:, None, None] * roi
        np.exp(z, out=z)
        share = rng.uniform(0.05, 0.5, (H, M, 1)).astype(np.float32)
        z *= share / z.sum(axis=-1, keepdims=True)
        out[l] = f32_to_bf16_bits(z)

    if M > 0:
        with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
            list(ex.map(layer, range(L)))
    return out


def make_attention_batch(w: AttentionWorkload, B: int | None = None, lens=None, threads: int = 8, L=None, H=None,
                         N=None):
    """(attn, lens, attn_ref): attn = the samples' [L, H, M_b, N] blocks flattened and packed
    in sample order (uint16, 1-D), lens [B] int32, attn_ref [B, L, H, m_ref, N] uint16."""
    B = B or w.B
    lens = attention_lens(w, B) if lens is None else np.asarray(lens, dtype=np.int32)
    blocks = [make_attention(w, b, int(lens[b]), False, L, H, N, threads).reshape(-1) for b in range(B)]
    attn = np.concatenate(blocks) if blocks else np.zeros(0, np.uint16)
    ref = np.stack([make_attention(w, b, w.m_ref, True, L, H, N, threads) for b in range(B)])
    return attn, lens, ref


# ----------------------------------------------------------------------------- ragged batches

@dataclasses.dataclass(frozen=True)
class RaggedWorkload:
    """Variable-resolution images (Qwen2.5-VL-style dynamic token counts) in a padded batch:
    image b has n_valid[b] tokens on its own rows x cols grid, at most n_max."""
    name: str
    config_id: int
    B: int
    n_max: int
    n_lo: int           # smallest token count drawn
    D: int
    centroids: int      # per image, on an 8 x 8 block grid over its token grid
    noise: float
    m_lo: int
    m_hi: int
    K: int


RAGGED_WORKLOADS = {
    # Qwen2.5-VL-7B width (D = 3584), up to 1280 visual tokens per image, keep 128
    "c5": RaggedWorkload("c5_ragged16_nmax1280_k128", 5, 16, 1280, 640, 3584, 64, 0.3, 16, 128, 128),
}


def make_ragged_image(w: RaggedWorkload, image: int, D: int | None = None):
    """(bits [n_max, D], n_valid): a rows x cols token grid (rows in [20, 32], n_valid =
    rows * cols drawn near U[n_lo, n_max]) of clustered features (centroid of the token's
    block on an 8 x 8 block grid + N(0, noise^2)); the padding rows after n_valid hold
    unrelated N(0, 5^2) values, which no result may depend on."""
    D = D or w.D
    rng = np.random.Generator(np.random.PCG64(1000 * w.config_id + image))
    rows = int(rng.integers(20, 33))
    target = int(rng.integers(w.n_lo, w.n_max + 1))
    cols = max(1, min(target // rows, w.n_max // rows))
    nv = rows * cols
    r = np.arange(rows)[:, None] * 8 // rows
    c = np.arange(cols)[None, :] * 8 // cols
    cid = (r * 8 + c).reshape(-1) % w.centroids
    cent = rng.standard_normal((w.centroids, D), dtype=np.float32)
    x = np.empty((w.n_max, D), dtype=np.float32)
    x[:nv] = cent[cid] + rng.standard_normal((nv, D), dtype=np.float32) * np.float32(w.noise)
    x[nv:] = rng.standard_normal((w.n_max - nv, D), dtype=np.float32) * np.float32(5.0)
    return f32_to_bf16_bits(x), nv


def make_ragged_batch(w: RaggedWorkload, B: int | None = None, threads: int = 8, D: int | None = None):
    """(vis [B, n_max, D] u16, text [sum(lens), D] u16, lens [B] int32, n_valid [B] int32)."""
    B = B or w.B
    D = D or w.D
    rng = np.random.Generator(np.random.PCG64(1000 * w.config_id + 999_999))
    lens = rng.integers(w.m_lo, w.m_hi + 1, size=B).astype(np.int32)
    vis = np.empty((B, w.n_max, D), dtype=np.uint16)
    nv = np.empty(B, dtype=np.int32)
    texts = [None] * B

    def one(b):
        vis[b], nv[b] = make_ragged_image(w, b, D)
        trng = np.random.Generator(np.random.PCG64(1000 * w.config_id + b + 1_000_000))
        texts[b] = f32_to_bf16_bits(trng.standard_normal((int(lens[b]), D), dtype=np.float32))

    with ThreadPoolExecutor(max_workers=max(1, threads)) as ex:
        list(ex.map(one, range(B)))
    return vis, np.concatenate(texts, axis=0), lens, nv
