"""The C-ABI library: it builds, loads without a GPU, exports every symbol that
include/map_gb300.h declares, and rejects bad arguments before touching the device.
CPU only: no compute call is made."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "map_gb300.h")


@pytest.fixture(scope="module")
def mb():
    from paper_2608_06411_gb300 import build_lib
    build_lib.build()
    from paper_2608_06411_gb300 import binding
    return binding


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(map_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported_and_bound(mb):
    names = declared_functions()
    assert len(names) >= 14
    for n in names:
        assert hasattr(mb.lib, n), n
        assert n in mb.SIGNATURES, n


def test_config_default_and_strerror(mb):
    cfg = mb.default_config()
    assert (cfg.D, cfg.Dh, cfg.dp, cfg.rope_on, cfg.k0_abs) == (4096, 1024, 128, 1, -1)
    assert abs(cfg.lam - 1.0) < 1e-7 and abs(cfg.k0_frac - 0.5) < 1e-7 and abs(cfg.tau - 1e-5) < 1e-12
    assert mb.lib.map_strerror(mb.MAP_EINVAL) == b"invalid argument"
    assert mb.lib.map_strerror(mb.MAP_ETIMEOUT) == b"device-side wait timed out"
    assert mb.lib.map_config_default(None) == mb.MAP_EINVAL


def test_bad_arguments_are_rejected_on_the_host(mb):
    lib = mb.lib
    h = ctypes.c_void_p()
    bad = mb.default_config()
    bad.dp = 96
    w = mb.MapWeights(*([ctypes.c_void_p(16)] * 10))
    assert lib.map_init(ctypes.byref(bad), ctypes.byref(w), ctypes.byref(h)) == mb.MAP_EINVAL
    assert not h.value
    bad = mb.default_config()
    bad.D = 100
    assert lib.map_init(ctypes.byref(bad), ctypes.byref(w), ctypes.byref(h)) == mb.MAP_EINVAL
    good = mb.default_config()
    w0 = mb.MapWeights()
    assert lib.map_init(ctypes.byref(good), ctypes.byref(w0), ctypes.byref(h)) == mb.MAP_EINVAL
    assert lib.map_init(ctypes.byref(good), ctypes.byref(w), None) == mb.MAP_EINVAL
    lens = (ctypes.c_int32 * 1)(4)
    assert lib.map_score(None, 16, 16, lens, 1, 8, 16, None) == mb.MAP_EINVAL
    assert lib.map_select(None, 16, 16, 1, 8, 2, 16, None, None) == mb.MAP_EINVAL
    assert lib.map_gather(None, 16, 16, 1, 8, 2, 16, None) == mb.MAP_EINVAL
    assert lib.map_prune(None, 16, 16, lens, 1, 8, 2, 16, 16, None, None) == mb.MAP_EINVAL
    assert lib.map_status(None, None) == mb.MAP_EINVAL
    assert lib.map_get_counters(None, None) == mb.MAP_EINVAL
    lib.map_destroy(None)


def test_qcts_bad_arguments_are_rejected_on_the_host(mb):
    lib = mb.lib
    lens = (ctypes.c_int32 * 2)(3, 4)
    neg = (ctypes.c_int32 * 2)(3, -1)
    f = 256   # a non-null stand-in; nothing is dereferenced or launched on an argument error
    assert lib.map_qcts(None, lens, f, 2, 2, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, None, f, 2, 2, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, lens, f, 2, 2, 4, 2, 8, None, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, lens, f, 0, 2, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, lens, f, 2, 0, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, lens, f, 2, 2, 0, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, lens, f, 2, 2, 4, 2, 0, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f, neg, f, 2, 2, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_qcts(f + 1, lens, f, 2, 2, 4, 2, 8, f, f, f, f, None, None) == mb.MAP_EINVAL


def test_assemble_bad_arguments_are_rejected_on_the_host(mb):
    lib = mb.lib
    lens = (ctypes.c_int32 * 1)(3)
    neg = (ctypes.c_int32 * 1)(-1)
    f = 256
    assert lib.map_assemble(None, f, f, f, lens, 1, 8, 2, 0, f, f, None) == mb.MAP_EINVAL
    assert lib.map_assemble(f, f, f, f, neg, 1, 8, 2, 0, f, f, None) == mb.MAP_EINVAL
    assert lib.map_assemble(f, f, f, f, lens, 1, 8, 9, 0, f, f, None) == mb.MAP_EINVAL
    assert lib.map_assemble(f, f, f, f, lens, 0, 8, 2, 0, f, f, None) == mb.MAP_EINVAL


def test_ragged_bad_arguments_are_rejected_on_the_host(mb):
    lib = mb.lib
    lens = (ctypes.c_int32 * 2)(3, 4)
    nv_ok = (ctypes.c_int32 * 2)(8, 5)
    nv_big = (ctypes.c_int32 * 2)(9, 5)
    nv_zero = (ctypes.c_int32 * 2)(8, 0)
    f = 256
    assert lib.map_score_ragged(None, f, f, lens, nv_ok, 2, 8, f, None) == mb.MAP_EINVAL
    assert lib.map_score_ragged(f, f, f, lens, None, 2, 8, f, None) == mb.MAP_EINVAL
    assert lib.map_select_ragged(f, f, f, None, 2, 8, 2, f, None, None) == mb.MAP_EINVAL
    assert lib.map_prune_ragged(f, f, f, lens, None, 2, 8, 2, f, f, None, None) == mb.MAP_EINVAL
    # sizes checked before the context is touched
    assert lib.map_prune_ragged(f, f, f, lens, nv_big, 2, 8, 2, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_prune_ragged(f, f, f, lens, nv_zero, 2, 8, 2, f, f, None, None) == mb.MAP_EINVAL
    assert lib.map_prune_ragged(f, f, f, lens, nv_ok, 2, 8, 6, f, f, None, None) == mb.MAP_EINVAL


def test_select_noalloc_bad_arguments_are_rejected_on_the_host(mb):
    lib = mb.lib
    f = 256   # a non-null, 16-byte aligned stand-in; the context is not touched on these errors
    assert lib.map_select_noalloc(None, f, f, 1, 8, 2, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, None, f, 1, 8, 2, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, None, 1, 8, 2, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f, 0, 8, 2, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f, 1, 0, 0, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f, 1, 8, 9, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f, 1, 8, -1, f, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f, 1, 8, 2, None, None, None) == mb.MAP_EINVAL
    assert lib.map_select_noalloc(f, f, f + 8, 1, 8, 2, f, None, None) == mb.MAP_EINVAL   # misaligned features
    assert lib.map_select_noalloc(f, f, f, 1, 16385, 2, f, None, None) == mb.MAP_EUNSUPPORTED
    assert lib.map_select_noalloc(f, f, f, 1, 8000, 4097, f, None, None) == mb.MAP_EUNSUPPORTED
    assert lib.map_select_noalloc(f, f, f, 1, 8, 0, None, None, None) == mb.MAP_OK          # k = 0: nothing to do
