"""Predictor weights on disk: one file, a JSON header and the bf16 bit patterns.

A trained predictor (the paper trains it by distillation; `map_distill_grad` gives the
gradients) is stored and reloaded with this format, then handed to `map_init` (through
`binding.Context`), which accepts host or device pointers.

File layout (little-endian):
  bytes 0-7     magic b"MAPW" and the format version (uint32, 1)
  bytes 8-15    header length H in bytes (uint64)
  bytes 16..    H bytes of UTF-8 JSON:
                  {"D": .., "Dh": .., "dp": .., "dtype": "bf16",
                   "tensors": [{"name": .., "shape": [..], "offset": .., "nbytes": ..}, ...]}
  then          the data section: each tensor's bf16 bits in row-major order, starting at
                its offset (a multiple of 16) from the start of the data section, which
                itself starts at the next multiple of 16 after the header.
The ten tensors are the predictor's weights in PyTorch Linear layout [out, in]: the question
MLP wT1 [Dh, D], bT1 [Dh], wT2 [Dh, Dh], bT2 [Dh]; the query projection wQ [dp, Dh]; the
visual MLP wV1 [Dh, D], bV1 [Dh], wV2 [Dh, Dh], bV2 [Dh]; the key projection wK [dp, Dh].
Loading checks the magic, the version, every name and shape against the stated widths, and
that every tensor lies inside the file; anything else raises ValueError.
"""
from __future__ import annotations

import json
import struct

import numpy as np

WEIGHT_NAMES = ("wT1", "bT1", "wT2", "bT2", "wQ", "wV1", "bV1", "wV2", "bV2", "wK")
MAGIC = b"MAPW"
VERSION = 1


def expected_shapes(D: int, Dh: int, dp: int) -> dict:
    """Shape of every predictor tensor for input width D, MLP width Dh and head width dp."""
    return {"wT1": (Dh, D), "bT1": (Dh,), "wT2": (Dh, Dh), "bT2": (Dh,), "wQ": (dp, Dh),
            "wV1": (Dh, D), "bV1": (Dh,), "wV2": (Dh, Dh), "bV2": (Dh,), "wK": (dp, Dh)}


def _round16(n: int) -> int:
    return (n + 15) // 16 * 16


def _bits(a) -> np.ndarray:
    """bf16 bit patterns as a C-contiguous uint16 array (uint16 or int16 input)."""
    a = np.asarray(a)
    if a.dtype not in (np.uint16, np.int16):
        raise ValueError(f"weights must be bf16 bit patterns (uint16 or int16), got {a.dtype}")
    return np.ascontiguousarray(a).view(np.uint16)


def save_weights(path: str, weights: dict, D: int, Dh: int, dp: int) -> None:
    """Writes the ten predictor tensors (bf16 bits, host arrays) with their widths."""
    shapes = expected_shapes(D, Dh, dp)
    entries, blobs, off = [], [], 0
    for name in WEIGHT_NAMES:
        if name not in weights:
            raise ValueError(f"missing weight {name}")
        a = _bits(weights[name])
        if a.shape != shapes[name]:
            raise ValueError(f"{name}: shape {a.shape}, expected {shapes[name]} for D={D}, Dh={Dh}, dp={dp}")
        entries.append({"name": name, "shape": list(a.shape), "offset": off, "nbytes": int(a.nbytes)})
        blobs.append((off, a))
        off = _round16(off + a.nbytes)
    header = json.dumps({"D": D, "Dh": Dh, "dp": dp, "dtype": "bf16", "tensors": entries}).encode()
    data_start = _round16(16 + len(header))
    with open(path, "wb") as f:
        f.write(MAGIC + struct.pack("<I", VERSION) + struct.pack("<Q", len(header)))
        f.write(header)
        f.write(b"\0" * (data_start - 16 - len(header)))
        pos = 0
        for o, a in blobs:
            f.write(b"\0" * (o - pos))
            f.write(a.tobytes())
            pos = o + a.nbytes


def load_weights(path: str):
    """Returns (weights {name: uint16 [shape]}, dims {"D", "Dh", "dp"})."""
    with open(path, "rb") as f:
        raw = f.read()
    if len(raw) < 16 or raw[:4] != MAGIC:
        raise ValueError(f"{path}: not a predictor weight file")
    version, = struct.unpack("<I", raw[4:8])
    if version != VERSION:
        raise ValueError(f"{path}: format version {version}, this reader takes {VERSION}")
    hlen, = struct.unpack("<Q", raw[8:16])
    if 16 + hlen > len(raw):
        raise ValueError(f"{path}: header runs past the end of the file")
    try:
        head = json.loads(raw[16:16 + hlen].decode())
        D, Dh, dp = int(head["D"]), int(head["Dh"]), int(head["dp"])
        tensors = {t["name"]: t for t in head["tensors"]}
    except (ValueError, KeyError, TypeError) as e:
        raise ValueError(f"{path}: malformed header ({e})") from None
    if head.get("dtype") != "bf16":
        raise ValueError(f"{path}: dtype {head.get('dtype')!r}, expected 'bf16'")
    if min(D, Dh, dp) < 1:
        raise ValueError(f"{path}: widths D={D}, Dh={Dh}, dp={dp} must be positive")
    if sorted(tensors) != sorted(WEIGHT_NAMES):
        raise ValueError(f"{path}: tensors {sorted(tensors)}, expected {sorted(WEIGHT_NAMES)}")
    shapes = expected_shapes(D, Dh, dp)
    data_start = _round16(16 + hlen)
    out = {}
    for name in WEIGHT_NAMES:
        t = tensors[name]
        shape = tuple(int(x) for x in t["shape"])
        if shape != shapes[name]:
            raise ValueError(f"{path}: {name} has shape {shape}, expected {shapes[name]}")
        off, nbytes = int(t["offset"]), int(t["nbytes"])
        if nbytes != 2 * int(np.prod(shape)) or off < 0 or off % 16:
            raise ValueError(f"{path}: {name} has offset {off} and {nbytes} bytes for shape {shape}")
        lo = data_start + off
        if lo + nbytes > len(raw):
            raise ValueError(f"{path}: {name} runs past the end of the file")
        out[name] = np.frombuffer(raw, dtype=np.uint16, count=nbytes // 2, offset=lo).reshape(shape).copy()
    return out, {"D": D, "Dh": Dh, "dp": dp}
