"""Hand-worked examples of Eq. 4 and the paper's stated workload facts (tests/golden/)."""
import json
import os

import numpy as np
import pytest

from oracle import map_oracle as O
from paper_2608_06411_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


CASES = _load("hand_selection.json")["cases"]


@pytest.mark.parametrize("case", CASES, ids=[c["name"] for c in CASES])
def test_hand_worked_selection(case):
    V = np.array(case["V"], dtype=np.float64)
    p = np.array(case["p"], dtype=np.float64)
    for lam, want in case["expect"].items():
        r = O.select(p, V, case["K"], case["K0"], lam=float(lam))
        assert r["picks"].tolist() == want, (lam, r["picks"])
        assert r["keep"].tolist() == sorted(want)
    if "margins" in case:
        r = O.select(p, V, case["K"], case["K0"], lam=1.0)
        np.testing.assert_allclose(r["margins"], case["margins"], rtol=1e-12)


def test_workload_shapes_follow_the_paper():
    g = _load("paper_workloads.json")
    c1, c0 = W.WORKLOADS["c1"], W.WORKLOADS["c0"]
    assert c1.N == g["llava_next_tokens"] and c0.N == g["llava15_tokens"]
    assert c1.K in g["llava_next_budgets"] and c0.K in g["llava15_budgets"]
    assert round(100 * c1.K / c1.N, 2) == g["llava_next_kept_fraction_percent"]
    c4 = W.WORKLOADS["c4"]
    assert round(100 * c4.K / c4.N, 2) == g["llava_next_kept_fraction_percent"]
    c3 = W.WORKLOADS["c3"]
    assert (c3.N, c3.K, c3.B) == (2880, 160, 64)
