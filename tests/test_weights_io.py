"""Predictor weight files: a round trip keeps every bit, widths and names; malformed files
are rejected with ValueError (CPU only)."""
import json
import struct

import numpy as np
import pytest

from paper_2608_06411_gb300 import weights_io as WIO
from paper_2608_06411_gb300 import workloads as W


def _weights(D=48, Dh=32, dp=16):
    dims = W.PredictorDims(D=D, Dh=Dh, dp=dp)
    return W.make_weights(dims, seed=5, bias_std=0.1), dims


def test_round_trip_keeps_every_bit(tmp_path):
    w, dims = _weights()
    p = tmp_path / "pred.mapw"
    WIO.save_weights(str(p), w, dims.D, dims.Dh, dims.dp)
    got, d = WIO.load_weights(str(p))
    assert d == {"D": dims.D, "Dh": dims.Dh, "dp": dims.dp}
    assert list(got) == list(WIO.WEIGHT_NAMES)
    for k in WIO.WEIGHT_NAMES:
        assert got[k].dtype == np.uint16 and got[k].flags["C_CONTIGUOUS"]
        np.testing.assert_array_equal(got[k], w[k])


def test_names_match_the_library_binding():
    mb = pytest.importorskip("paper_2608_06411_gb300.binding", exc_type=ImportError)
    assert tuple(mb.WEIGHT_NAMES) == WIO.WEIGHT_NAMES


def test_int16_views_are_accepted(tmp_path):
    w, dims = _weights()
    p = tmp_path / "pred.mapw"
    WIO.save_weights(str(p), {k: v.view(np.int16) for k, v in w.items()}, dims.D, dims.Dh, dims.dp)
    got, _ = WIO.load_weights(str(p))
    np.testing.assert_array_equal(got["wK"], w["wK"])


def test_data_offsets_are_16_byte_aligned(tmp_path):
    w, dims = _weights(D=40, Dh=24, dp=8)
    p = tmp_path / "pred.mapw"
    WIO.save_weights(str(p), w, dims.D, dims.Dh, dims.dp)
    raw = p.read_bytes()
    hlen, = struct.unpack("<Q", raw[8:16])
    head = json.loads(raw[16:16 + hlen])
    assert all(t["offset"] % 16 == 0 for t in head["tensors"])
    assert len(raw) >= (16 + hlen + 15) // 16 * 16 + head["tensors"][-1]["offset"] + head["tensors"][-1]["nbytes"]


def test_save_rejects_wrong_shapes_and_types(tmp_path):
    w, dims = _weights()
    p = str(tmp_path / "x.mapw")
    with pytest.raises(ValueError, match="shape"):
        WIO.save_weights(p, {**w, "wQ": w["wK"][:, :-1]}, dims.D, dims.Dh, dims.dp)
    with pytest.raises(ValueError, match="missing"):
        WIO.save_weights(p, {k: v for k, v in w.items() if k != "bV2"}, dims.D, dims.Dh, dims.dp)
    with pytest.raises(ValueError, match="bf16"):
        WIO.save_weights(p, {**w, "wK": w["wK"].astype(np.float32)}, dims.D, dims.Dh, dims.dp)


def _rewrite_header(raw: bytes, edit) -> bytes:
    hlen, = struct.unpack("<Q", raw[8:16])
    head = json.loads(raw[16:16 + hlen])
    edit(head)
    new = json.dumps(head).encode()
    data_start = (16 + hlen + 15) // 16 * 16
    pad = (16 + len(new) + 15) // 16 * 16 - 16 - len(new)
    return raw[:8] + struct.pack("<Q", len(new)) + new + b"\0" * pad + raw[data_start:]


@pytest.mark.parametrize("mutate,match", [
    (lambda raw: b"XXXX" + raw[4:], "not a predictor weight file"),
    (lambda raw: raw[:4] + struct.pack("<I", 9) + raw[8:], "version"),
    (lambda raw: raw[:-2], "past the end"),
    (lambda raw: raw[:20], "past the end|malformed"),
    (lambda raw: _rewrite_header(raw, lambda h: h.update(dp=h["dp"] + 1)), "shape"),
    (lambda raw: _rewrite_header(raw, lambda h: h.update(dtype="fp16")), "dtype"),
    (lambda raw: _rewrite_header(raw, lambda h: h["tensors"].pop()), "tensors"),
    (lambda raw: _rewrite_header(raw, lambda h: h["tensors"][0].update(offset=8)), "offset"),
])
def test_load_rejects_malformed_files(tmp_path, mutate, match):
    w, dims = _weights()
    p = tmp_path / "pred.mapw"
    WIO.save_weights(str(p), w, dims.D, dims.Dh, dims.dp)
    bad = tmp_path / "bad.mapw"
    bad.write_bytes(mutate(p.read_bytes()))
    with pytest.raises(ValueError, match=match):
        WIO.load_weights(str(bad))
