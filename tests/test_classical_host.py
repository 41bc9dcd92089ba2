"""Host-side checks of the classical-path measurement arm of bench.py (no GPU).

The classical path is the comparison whose traffic Eq. M_classical counts; these tests check
that it computes the same function as the oracle (on CPU tensors) and that the analytic model
reproduces the reduction factor the paper quotes for n = 32768, d_k = 64 (Section 8.2).
"""
import math
import os
import sys

import numpy as np
import pytest

torch = pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2606_07713_gb300 import inputs as I  # noqa: E402


def test_classical_step_matches_oracle(oracle):
    x = I.make_inputs(I.custom_config(2, 2, 37, 53, 16, 8, dtype="fp32", seed=5))
    q, k, v = (torch.from_numpy(a.astype(np.float64)) for a in (x.q, x.k, x.v))
    o = bench.classical_step(q, k, v, x.scale).numpy()
    ref = oracle.attn(x.q, x.k, x.v, x.scale)
    assert np.max(np.abs(o - ref)) <= 1e-12


def test_analytic_reduction_factor():
    s = I.AttnShape(1, 1, 32768, 32768, 64, 64)
    a = bench.analytic_traffic(s)
    n, d = 32768, 64
    assert a["M_moa_elements"] == 3 * n * d
    assert a["M_classical_elements"] == 3 * n * n + 3 * n * d + n
    # the paper's k ~ n / d_k = 512 for this case
    assert math.isclose(a["k_analytic"], 512.0, rel_tol=0.01)
