"""Property-based pins of the fp64 oracle (CPU only): for random tiny shapes, values and scales
(negative ones included), the oracle's output agrees with softmax(scale Q K^T) V evaluated
independently in 50-digit decimal arithmetic, and its rows keep the properties Eq. attention
fixes for any input."""
import math

import numpy as np
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402

import oracle_pins  # noqa: E402

SHAPES = st.tuples(st.integers(1, 4), st.integers(1, 6), st.integers(1, 6), st.integers(1, 4))


def _draw(shape, seed, spread):
    nq, nk, dk, dv = shape
    r = np.random.default_rng(seed)
    f32 = lambda a: np.asarray(a, dtype=np.float32)
    return (f32(r.normal(size=(nq, dk)) * spread), f32(r.normal(size=(nk, dk)) * spread),
            f32(r.normal(size=(nk, dv))))


@settings(max_examples=40, deadline=None)
@given(shape=SHAPES, seed=st.integers(0, 2**31 - 1), spread=st.sampled_from([0.1, 1.0, 3.0]),
       scale=st.floats(-2.0, 2.0, allow_nan=False, allow_infinity=False))
def test_oracle_matches_decimal_bruteforce(oracle, shape, seed, spread, scale):
    Q, K, V = _draw(shape, seed, spread)
    ref = oracle_pins.decimal_attention(Q, K, V, scale)
    got = oracle.attn(Q, K, V, scale)
    err = np.max(np.abs(got - ref)) / max(1e-300, np.max(np.abs(ref)))
    assert err <= 1e-12, (shape, seed, spread, scale, err)


@settings(max_examples=40, deadline=None)
@given(shape=SHAPES, seed=st.integers(0, 2**31 - 1), spread=st.sampled_from([0.1, 1.0, 3.0]),
       scale=st.floats(-2.0, 2.0, allow_nan=False, allow_infinity=False))
def test_oracle_rows_are_convex_combinations(oracle, shape, seed, spread, scale):
    """Each output row is a convex combination of the value rows: it lies in their per-column
    range, and with V = 1 it is exactly 1."""
    Q, K, V = _draw(shape, seed, spread)
    O = oracle.attn(Q, K, V, scale)
    lo, hi = V.astype(np.float64).min(axis=0), V.astype(np.float64).max(axis=0)
    tol = 1e-12 * (1.0 + np.abs(V).max())
    assert np.all(O >= lo - tol) and np.all(O <= hi + tol)
    ones = np.ones_like(V)
    assert np.max(np.abs(oracle.attn(Q, K, ones, scale) - 1.0)) <= 1e-14


@settings(max_examples=30, deadline=None)
@given(shape=SHAPES, seed=st.integers(0, 2**31 - 1), shift=st.floats(-50.0, 50.0))
def test_oracle_ignores_a_common_score_shift(oracle, shape, seed, shift):
    """Adding the same constant to every score of a row leaves the row unchanged: a key feature
    fixed at 1 and a query feature set to shift/scale add exactly `shift` to each score."""
    nq, nk, dk, dv = shape
    Q, K, V = _draw((nq, nk, dk + 1, dv), seed, 1.0)
    scale = 1.0 / math.sqrt(dk + 1)
    K[:, 0] = 1.0
    Qa, Qb = Q.copy(), Q.copy()
    Qa[:, 0] = 0.0
    Qb[:, 0] = np.float32(shift / scale)
    oa, ob = oracle.attn(Qa, K, V, scale), oracle.attn(Qb, K, V, scale)
    assert np.max(np.abs(oa - ob)) <= 1e-12 * (1.0 + np.abs(V).max())
