"""Oracle runs for whole-batch GPU parity checks, spread over a pool of host processes, and
the per-configuration record of how the GPU selection compared with the oracle.

The pool uses the "spawn" start method (a process forked after CUDA was initialised can
hang) and one BLAS thread per worker.  Workers rebuild each image's inputs from the seeded
generators (workload name, image index), so only scores and pick lists cross processes.
No torch import here: the workers never touch the GPU."""
from __future__ import annotations

import multiprocessing
import os
from concurrent.futures import ProcessPoolExecutor

import numpy as np

from oracle import map_oracle as O
from oracle import parity as P
from paper_2608_06411_gb300 import workloads as W

_POOL = None
_WEIGHTS = {}

# (config label, images checked, images identical to the oracle's pick order, images with
# at least one sub-margin step, total sub-margin steps, worst score relative error)
SELECTION_STATS: list = []


def pool() -> ProcessPoolExecutor:
    global _POOL
    if _POOL is None:
        saved = {v: os.environ.get(v) for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")}
        for v in saved:
            os.environ[v] = "1"
        try:
            _POOL = ProcessPoolExecutor(max_workers=max(1, min(16, os.cpu_count() or 1)),
                                        mp_context=multiprocessing.get_context("spawn"))
        finally:
            for v, x in saved.items():
                if x is None:
                    os.environ.pop(v, None)
                else:
                    os.environ[v] = x
    return _POOL


def shutdown():
    global _POOL
    if _POOL is not None:
        _POOL.shutdown(wait=True, cancel_futures=True)
        _POOL = None


def _weights(D: int, seed: int = 7) -> dict:
    key = (D, seed)
    if key not in _WEIGHTS:
        _WEIGHTS[key] = W.make_weights(W.PredictorDims(D=D), seed=seed)
    return _WEIGHTS[key]


def oracle_scores(wl_name: str, b: int, m: int) -> np.ndarray:
    """Eq. 3 for image b of the workload with its m question tokens (float64 [N])."""
    wl = W.WORKLOADS[wl_name]
    vis = W.make_image(wl, b)
    text = W.make_text(wl, b, m)
    return O.map_score(text, vis[None], [m], _weights(wl.D))[0]


def oracle_check(wl_name: str, b: int, p32: np.ndarray, K: int, K0: int, order, keep, lam: float = 1.0,
                 tau: float = 1e-5) -> dict:
    """check_selection of the GPU's pick order for image b on the fp32 scores it was given."""
    wl = W.WORKLOADS[wl_name]
    V = O.bf16_bits_to_f64(W.make_image(wl, b))
    return P.check_selection(np.asarray(p32, dtype=np.float32).astype(np.float64), V, K, K0, order, keep,
                             lam=lam, tau=tau)


def record(label: str, reps: list, score_err: float | None = None):
    """Adds one configuration's selection outcome to the session summary."""
    identical = sum(1 for r in reps if r["identical"])
    with_sub = sum(1 for r in reps if r["sub_margin_steps"] > 0)
    steps = sum(int(r["sub_margin_steps"]) for r in reps)
    SELECTION_STATS.append((label, len(reps), identical, with_sub, steps, score_err))
