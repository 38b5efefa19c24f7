"""The host process pool that the whole-batch GPU parity tests use: a spawned worker
returns exactly what the oracle returns in this process.  CPU only."""
import numpy as np

import _oracle_pool as OP
from oracle import map_oracle as O
from paper_2608_06411_gb300 import workloads as W


def test_pool_workers_reproduce_the_oracle():
    wl = W.WORKLOADS["c0"]
    ex = OP.pool()
    f = ex.submit(OP.oracle_scores, "c0", 3, 5)
    vis = W.make_image(wl, 3)
    w = W.make_weights(W.PredictorDims(D=wl.D))
    p = O.map_score(W.make_text(wl, 3, 5), vis[None], [5], w)[0]
    np.testing.assert_array_equal(f.result(), p)
    p32 = p.astype(np.float32)
    r = O.select(p32.astype(np.float64), O.bf16_bits_to_f64(vis), wl.K, O.resolve_k0(wl.K))
    rep = ex.submit(OP.oracle_check, "c0", 3, p32, wl.K, O.resolve_k0(wl.K), r["picks"], r["keep"]).result()
    assert rep["ok"] and rep["identical"]
    OP.shutdown()
