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


@settings(max_examples=15, deadline=None)
@given(shape=st.tuples(st.integers(1, 3), st.integers(1, 4), st.integers(1, 3), st.integers(1, 3)),
       seed=st.integers(0, 2**31 - 1), scale=st.floats(-1.5, 1.5, allow_nan=False))
def test_backward_oracle_matches_decimal_central_differences(oracle, shape, seed, scale):
    """Every entry of dQ, dK and dV from the backward oracle against a central difference of
    L = sum(dO * O) in 60-digit decimal arithmetic, on random tiny inputs and scales."""
    import decimal
    nq, nk, dk, dv = shape
    r = np.random.default_rng(seed)
    f32 = lambda a: np.asarray(a, dtype=np.float32)
    Q, K = f32(r.normal(size=(nq, dk)) * 1.5), f32(r.normal(size=(nk, dk)))
    V, G = f32(r.normal(size=(nk, dv))), f32(r.normal(size=(nq, dv)))
    grads = oracle.attn_bwd(Q, K, V, G, scale)
    ctx = decimal.Context(prec=60)
    D = lambda x: decimal.Decimal(float(x))
    mats = [[[D(x) for x in row] for row in M] for M in (Q, K, V)]
    g = [[D(x) for x in row] for row in G]
    sc, h = D(scale), decimal.Decimal("1e-12")
    for which, grad in enumerate(grads):
        M = mats[which]
        for a in range(len(M)):
            for b in range(len(M[0])):
                keep = M[a][b]
                M[a][b] = keep + h
                lp = oracle_pins._decimal_loss(mats[0], mats[1], mats[2], g, sc, ctx)
                M[a][b] = keep - h
                lm = oracle_pins._decimal_loss(mats[0], mats[1], mats[2], g, sc, ctx)
                M[a][b] = keep
                fd = float(ctx.divide(ctx.subtract(lp, lm), 2 * h))
                assert abs(grad[a, b] - fd) <= 1e-12 * max(1.0, abs(fd)), (shape, which, a, b)
