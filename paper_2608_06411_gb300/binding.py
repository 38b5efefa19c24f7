"""Thin ctypes binding of libmap_gb300 (include/map_gb300.h): argument marshalling only.

Every step of the pruning path runs in the CUDA library; this module passes tensor
pointers, sizes and the current CUDA stream through and turns error codes into
exceptions.  Importing it loads the library and raises ImportError if it is missing:
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_double, c_float, c_int, c_int32, c_longlong, c_void_p

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libmap_gb300.so")

MAP_OK, MAP_EINVAL, MAP_ENOMEM, MAP_ECUDA, MAP_ETIMEOUT, MAP_EUNSUPPORTED, MAP_EINTERNAL = 0, -1, -2, -3, -4, -5, -6
K_GEMM_FV1, K_GEMM_FV2, K_GEMM_WK, K_GEMM_TEXT, K_SCORES, K_SELECT, K_GATHER = range(7)
EPI_GELU_BF16, EPI_BIAS_BF16, EPI_F32 = 0, 1, 3

WEIGHT_NAMES = ("wT1", "bT1", "wT2", "bT2", "wQ", "wV1", "bV1", "wV2", "bV2", "wK")


class MapConfig(ctypes.Structure):
    _fields_ = [("D", c_int), ("Dh", c_int), ("dp", c_int), ("rope_theta", c_float), ("rope_on", c_int),
                ("k0_frac", c_float), ("k0_abs", c_int), ("lam", c_float), ("tau", c_float)]


class MapWeights(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in WEIGHT_NAMES]


class MapGrads(ctypes.Structure):
    _fields_ = [(n, c_void_p) for n in WEIGHT_NAMES]


class MapCounters(ctypes.Structure):
    _fields_ = [("launches", c_longlong), ("select_rounds", c_longlong), ("gram_rows", c_longlong)]


# Every symbol the header declares, with its ctypes signature.
SIGNATURES = {
    "map_config_default": (c_int, [POINTER(MapConfig)]),
    "map_init": (c_int, [POINTER(MapConfig), POINTER(MapWeights), POINTER(c_void_p)]),
    "map_score": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_int, c_int, c_void_p, c_void_p]),
    "map_select": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p, c_void_p]),
    "map_select_noalloc": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p,
                                   c_void_p]),
    "map_gather": (c_int, [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p, c_void_p]),
    "map_qcts": (c_int, [c_void_p, POINTER(c_int32), c_void_p, c_int, c_int, c_int, c_int, c_int, c_void_p, c_void_p,
                         c_void_p, c_void_p, c_void_p, c_void_p]),
    "map_assemble": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_int, c_int, c_int, c_int,
                             c_void_p, c_void_p, c_void_p]),
    "map_score_ragged": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), POINTER(c_int32), c_int, c_int,
                                 c_void_p, c_void_p]),
    "map_select_ragged": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_int, c_int, c_int, c_void_p,
                                  c_void_p, c_void_p]),
    "map_prune_ragged": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), POINTER(c_int32), c_int, c_int,
                                 c_int, c_void_p, c_void_p, c_void_p, c_void_p]),
    "map_assemble_ragged": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, POINTER(c_int32), POINTER(c_int32),
                                    c_int, c_int, c_int, c_int, c_void_p, c_void_p, c_void_p]),
    "map_distill_grad": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_void_p, c_int, c_int, c_void_p,
                                 POINTER(MapGrads), c_void_p]),
    "map_prune": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_int, c_int, c_int, c_void_p,
                          c_void_p, c_void_p, c_void_p]),
    "map_status": (c_int, [c_void_p, c_void_p]),
    "map_destroy": (None, [c_void_p]),
    "map_strerror": (ctypes.c_char_p, [c_int]),
    "map_get_counters": (c_int, [c_void_p, POINTER(MapCounters)]),
    "map_set_timing": (c_int, [c_void_p, c_int]),
    "map_set_wait_limit": (c_int, [c_void_p, c_longlong]),
    "map_read_timing": (c_int, [c_void_p, c_int, POINTER(c_double), POINTER(c_longlong)]),
    "map_linear": (c_int, [c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_void_p]),
    "map_score_debug": (c_int, [c_void_p, c_void_p, c_void_p, POINTER(c_int32), c_int, c_int, c_void_p, c_void_p,
                                c_void_p, c_void_p]),
}


def _load() -> ctypes.CDLL:
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is not built; run __graft_entry__.build() (nvcc, sm_103a)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


lib = _load()


class MapError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {lib.map_strerror(code).decode()} ({code})")


def _check(rc: int, where: str) -> None:
    if rc != MAP_OK:
        raise MapError(rc, where)


def _ptr(t) -> c_void_p:
    if t is None:
        return c_void_p(None)
    if isinstance(t, torch.Tensor):
        if not t.is_contiguous():
            raise ValueError("tensors passed to libmap_gb300 must be contiguous")
        return c_void_p(t.data_ptr())
    if isinstance(t, np.ndarray):
        if not t.flags["C_CONTIGUOUS"]:
            raise ValueError("arrays passed to libmap_gb300 must be C-contiguous")
        return c_void_p(t.ctypes.data)
    raise TypeError(f"unsupported buffer type {type(t)}")


def _stream(stream=None) -> c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return c_void_p(s.cuda_stream)


def _lens(lens) -> tuple:
    arr = np.ascontiguousarray(np.asarray(lens, dtype=np.int32))
    return arr, arr.ctypes.data_as(POINTER(c_int32))


def default_config() -> MapConfig:
    cfg = MapConfig()
    _check(lib.map_config_default(ctypes.byref(cfg)), "map_config_default")
    return cfg


class Context:
    """One library context (weights copied in at construction)."""

    def __init__(self, weights: dict, D: int, Dh: int, dp: int, rope_theta: float = 10000.0, rope_on: bool = True,
                 k0_frac: float = 0.5, k0_abs: int = -1, lam: float = 1.0, tau: float = 1e-5):
        self.cfg = MapConfig(D, Dh, dp, rope_theta, int(bool(rope_on)), k0_frac, k0_abs, lam, tau)
        keep = [np.ascontiguousarray(weights[n]) if isinstance(weights[n], np.ndarray) else weights[n].contiguous()
                for n in WEIGHT_NAMES]
        w = MapWeights(*[_ptr(t) for t in keep])
        h = c_void_p()
        _check(lib.map_init(ctypes.byref(self.cfg), ctypes.byref(w), ctypes.byref(h)), "map_init")
        self.h = h

    def close(self) -> None:
        if self.h:
            lib.map_destroy(self.h)
            self.h = c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the path -----------------------------------------------------------------------
    def score(self, text, vis, lens, scores=None, stream=None):
        B, N = vis.shape[0], vis.shape[1]
        if scores is None:
            scores = torch.empty((B, N), dtype=torch.float32, device=vis.device)
        arr, lp = _lens(lens)
        _check(lib.map_score(self.h, _ptr(text), _ptr(vis), lp, B, N, _ptr(scores), _stream(stream)), "map_score")
        return scores

    def score_debug(self, text, vis, lens, stream=None):
        B, N = vis.shape[0], vis.shape[1]
        arr, lp = _lens(lens)
        scores = torch.empty((B, N), dtype=torch.float32, device=vis.device)
        q = torch.empty((int(arr.sum()), self.cfg.dp), dtype=torch.float32, device=vis.device)
        k = torch.empty((B * N, self.cfg.dp), dtype=torch.float32, device=vis.device)
        _check(lib.map_score_debug(self.h, _ptr(text), _ptr(vis), lp, B, N, _ptr(scores), _ptr(q), _ptr(k),
                                   _stream(stream)), "map_score_debug")
        return scores, q, k

    def select(self, scores, vis, k: int, keep=None, order=None, want_order: bool = True, stream=None):
        B, N = vis.shape[0], vis.shape[1]
        if keep is None:
            keep = torch.empty((B, k), dtype=torch.int32, device=vis.device)
        if order is None and want_order:
            order = torch.empty((B, k), dtype=torch.int32, device=vis.device)
        _check(lib.map_select(self.h, _ptr(scores), _ptr(vis), B, N, k, _ptr(keep), _ptr(order), _stream(stream)),
               "map_select")
        return keep, order

    def select_noalloc(self, scores, vis, k: int, keep, order=None, stream=None):
        """map_select_noalloc: the caller provides keep (and order) buffers; nothing is
        allocated during the call."""
        B, N = vis.shape[0], vis.shape[1]
        _check(lib.map_select_noalloc(self.h, _ptr(scores), _ptr(vis), B, N, k, _ptr(keep), _ptr(order),
                                      _stream(stream)), "map_select_noalloc")
        return keep, order

    def gather(self, vis, keep, out=None, stream=None):
        B, N, D = vis.shape
        k = keep.shape[1]
        if out is None:
            out = torch.empty((B, k, D), dtype=vis.dtype, device=vis.device)
        _check(lib.map_gather(self.h, _ptr(vis), _ptr(keep), B, N, k, _ptr(out), _stream(stream)), "map_gather")
        return out

    def assemble(self, vis, keep, text, lens, pos_offset: int = 0, seq=None, pos=None, stream=None):
        """map_assemble: per image, the kept tokens then the question tokens, with position ids."""
        B, N, D = vis.shape
        k = keep.shape[1]
        arr, lp = _lens(lens)
        rows = B * k + int(arr.sum())
        if seq is None:
            seq = torch.empty((rows, D), dtype=vis.dtype, device=vis.device)
        if pos is None:
            pos = torch.empty(rows, dtype=torch.int32, device=vis.device)
        _check(lib.map_assemble(self.h, _ptr(vis), _ptr(keep), _ptr(text), lp, B, N, k, pos_offset, _ptr(seq),
                                _ptr(pos), _stream(stream)), "map_assemble")
        return seq, pos

    # -- ragged batches (padded layout, n_valid tokens per image) ---------------------------
    def score_ragged(self, text, vis, lens, n_valid, scores=None, stream=None):
        B, N = vis.shape[0], vis.shape[1]
        if scores is None:
            scores = torch.empty((B, N), dtype=torch.float32, device=vis.device)
        arr, lp = _lens(lens)
        nva, nvp = _lens(n_valid)
        _check(lib.map_score_ragged(self.h, _ptr(text), _ptr(vis), lp, nvp, B, N, _ptr(scores), _stream(stream)),
               "map_score_ragged")
        return scores

    def select_ragged(self, scores, vis, n_valid, k: int, keep=None, order=None, want_order: bool = True,
                      stream=None):
        B, N = vis.shape[0], vis.shape[1]
        if keep is None:
            keep = torch.empty((B, k), dtype=torch.int32, device=vis.device)
        if order is None and want_order:
            order = torch.empty((B, k), dtype=torch.int32, device=vis.device)
        nva, nvp = _lens(n_valid)
        _check(lib.map_select_ragged(self.h, _ptr(scores), _ptr(vis), nvp, B, N, k, _ptr(keep), _ptr(order),
                                     _stream(stream)), "map_select_ragged")
        return keep, order

    def prune_ragged(self, text, vis, lens, n_valid, k: int, out, keep, scores=None, stream=None):
        B, N = vis.shape[0], vis.shape[1]
        arr, lp = _lens(lens)
        nva, nvp = _lens(n_valid)
        _check(lib.map_prune_ragged(self.h, _ptr(text), _ptr(vis), lp, nvp, B, N, k, _ptr(out), _ptr(keep),
                                    _ptr(scores), _stream(stream)), "map_prune_ragged")
        return out, keep

    def assemble_ragged(self, vis, keep, text, lens, n_valid, pos_offset: int = 0, seq=None, pos=None,
                        stream=None):
        B, N, D = vis.shape
        k = keep.shape[1]
        arr, lp = _lens(lens)
        nva, nvp = _lens(n_valid)
        rows = B * k + int(arr.sum())
        if seq is None:
            seq = torch.empty((rows, D), dtype=vis.dtype, device=vis.device)
        if pos is None:
            pos = torch.empty(rows, dtype=torch.int32, device=vis.device)
        _check(lib.map_assemble_ragged(self.h, _ptr(vis), _ptr(keep), _ptr(text), lp, nvp, B, N, k, pos_offset,
                                       _ptr(seq), _ptr(pos), _stream(stream)), "map_assemble_ragged")
        return seq, pos

    def distill_grad(self, text, vis, lens, teacher, grads=None, loss=None, stream=None):
        """map_distill_grad: (loss [1], {weight name: fp32 gradient}) on device tensors."""
        B, N = vis.shape[0], vis.shape[1]
        D, Dh, dp = self.cfg.D, self.cfg.Dh, self.cfg.dp
        shapes = {"wT1": (Dh, D), "bT1": (Dh,), "wT2": (Dh, Dh), "bT2": (Dh,), "wQ": (dp, Dh),
                  "wV1": (Dh, D), "bV1": (Dh,), "wV2": (Dh, Dh), "bV2": (Dh,), "wK": (dp, Dh)}
        if grads is None:
            grads = {n: torch.empty(shapes[n], dtype=torch.float32, device=vis.device) for n in WEIGHT_NAMES}
        if loss is None:
            loss = torch.empty(1, dtype=torch.float32, device=vis.device)
        g = MapGrads(*[_ptr(grads[n]) for n in WEIGHT_NAMES])
        arr, lp = _lens(lens)
        _check(lib.map_distill_grad(self.h, _ptr(text), _ptr(vis), lp, _ptr(teacher), B, N, _ptr(loss),
                                    ctypes.byref(g), _stream(stream)), "map_distill_grad")
        return loss, grads

    def prune(self, text, vis, lens, k: int, out, keep, scores=None, stream=None):
        """score + select + gather in one C call; buffers may be host (pinned or not) or device."""
        B, N = vis.shape[0], vis.shape[1]
        arr, lp = _lens(lens)
        _check(lib.map_prune(self.h, _ptr(text), _ptr(vis), lp, B, N, k, _ptr(out), _ptr(keep), _ptr(scores),
                             _stream(stream)), "map_prune")
        return out, keep

    # -- diagnostics and instrumentation -------------------------------------------------
    def linear(self, x, w, b, epi: int, out=None, stream=None):
        M, K = x.shape
        Nout = w.shape[0]
        if out is None:
            dt = torch.float32 if epi == EPI_F32 else torch.bfloat16
            out = torch.empty((M, Nout), dtype=dt, device=x.device)
        _check(lib.map_linear(self.h, _ptr(x), _ptr(w), _ptr(b), M, K, Nout, epi, _ptr(out), _stream(stream)),
               "map_linear")
        return out

    def status(self, stream=None) -> int:
        return lib.map_status(self.h, _stream(stream))

    def check(self, stream=None) -> None:
        _check(self.status(stream), "map_status")

    def counters(self) -> dict:
        c = MapCounters()
        _check(lib.map_get_counters(self.h, ctypes.byref(c)), "map_get_counters")
        return {"launches": c.launches, "select_rounds": c.select_rounds, "gram_rows": c.gram_rows}

    def set_wait_limit(self, ns: int) -> None:
        """Limit of the GEMM kernels' waits in ns (<= 0: the 2 s default); for tests."""
        _check(lib.map_set_wait_limit(self.h, int(ns)), "map_set_wait_limit")

    def set_timing(self, enable: bool) -> None:
        _check(lib.map_set_timing(self.h, int(bool(enable))), "map_set_timing")

    def read_timing(self, kid: int) -> tuple:
        ms, n = c_double(), c_longlong()
        _check(lib.map_read_timing(self.h, kid, ctypes.byref(ms), ctypes.byref(n)), "map_read_timing")
        return ms.value, n.value


def qcts(attn, lens, attn_ref, L: int, H: int, N: int, p=None, p_ref=None, js=None, teacher=None,
         teacher_p=None, want_teacher_p: bool = True, stream=None):
    """map_qcts: Question Contrastive Teacher Selection on device tensors.

    attn: packed bf16 (int16 storage) attention of the B samples ([L, H, lens[b], N] blocks
    in sample order); attn_ref: [B, L, H, M_ref, N].  Returns (p, p_ref, js, teacher,
    teacher_p); outputs not given are allocated here."""
    arr, lp = _lens(lens)
    B = int(arr.shape[0])
    M_ref = int(attn_ref.shape[3])
    dev = attn_ref.device
    if p is None:
        p = torch.empty((B, L, N), dtype=torch.float32, device=dev)
    if p_ref is None:
        p_ref = torch.empty((B, L, N), dtype=torch.float32, device=dev)
    if js is None:
        js = torch.empty((B, L), dtype=torch.float32, device=dev)
    if teacher is None:
        teacher = torch.empty(B, dtype=torch.int32, device=dev)
    if teacher_p is None and want_teacher_p:
        teacher_p = torch.empty((B, N), dtype=torch.float32, device=dev)
    _check(lib.map_qcts(_ptr(attn), lp, _ptr(attn_ref), M_ref, B, L, H, N, _ptr(p), _ptr(p_ref), _ptr(js),
                        _ptr(teacher), _ptr(teacher_p), _stream(stream)), "map_qcts")
    return p, p_ref, js, teacher, teacher_p
