"""Pins for the fp64 oracle: facts fixed by the paper or by mathematics.

Each check takes an oracle object (oracle.Oracle) and raises AssertionError if
the oracle disagrees with the fact.  test_oracle_pins.py runs them against the
real oracle; test_oracle_mutants.py runs them against deliberately broken
copies of the oracle to show that each plausible mistake fails at least one
pin.  None of these checks re-types the oracle's own formula: they use values
printed in the paper, closed forms, invariants and an independent 50-digit
decimal brute force.
"""
from __future__ import annotations

import decimal
import math

import numpy as np

from conftest import load_golden


def _rng(seed):
    return np.random.default_rng(seed)


def _f32(x):
    return np.asarray(x, dtype=np.float32)


# ----------------------------------------------------------------------------------------------
# 1. The paper's worked example (Section 5, Tables tab:attn_weights and tab:output; Appendix A)
# ----------------------------------------------------------------------------------------------
def pin_paper_example(o):
    g = load_golden("paper_example_n3_d4.txt")
    Q, K, V = _f32(g["Q"]), _f32(g["K"]), _f32(g["V"])
    w, out = o.weights(Q, K, V, 0.5)
    # Printed to 4 decimals from inputs that were themselves printed to 4 decimals.
    assert np.max(np.abs(w - g["W"])) <= 2e-4, w
    assert np.max(np.abs(out - g["O"])) <= 2e-4, out
    assert np.max(np.abs(w.sum(axis=1) - 1.0)) <= 1e-12
    # Appendix A, row 0: scaled scores x, z = x - max x, e^z and their sum.
    x0 = o.scores(Q, K, 0.5)[0]
    assert np.max(np.abs(x0 - g["X0"][0])) <= 2e-4, x0
    z0 = x0 - x0.max()
    assert np.max(np.abs(z0 - g["Z0"][0])) <= 2e-4
    # e^z and Z follow from the oracle's weights: w = e^z / Z with max e^z = 1.
    e0 = w[0] / w[0].max()
    assert np.max(np.abs(e0 - g["E0"][0])) <= 2e-4, e0
    assert abs(1.0 / w[0].max() - g["DEN0"][0, 0]) <= 2e-4


# ----------------------------------------------------------------------------------------------
# 2. Independent brute force: 50-digit decimal arithmetic on tiny inputs
# ----------------------------------------------------------------------------------------------
def decimal_attention(Q, K, V, scale):
    """softmax(scale Q K^T) V evaluated in 50-digit decimal arithmetic (no max shift needed)."""
    ctx = decimal.Context(prec=50)
    D = lambda x: decimal.Decimal(float(x))
    n, dk = Q.shape
    nk, dv = V.shape
    sc = D(scale)
    out = np.zeros((n, dv))
    for i in range(n):
        ex = []
        for k in range(nk):
            s = decimal.Decimal(0)
            for j in range(dk):
                s = ctx.add(s, ctx.multiply(D(Q[i, j]), D(K[k, j])))
            ex.append(ctx.exp(ctx.multiply(s, sc)))
        tot = decimal.Decimal(0)
        for e in ex:
            tot = ctx.add(tot, e)
        for c in range(dv):
            acc = decimal.Decimal(0)
            for k in range(nk):
                acc = ctx.add(acc, ctx.multiply(ctx.divide(ex[k], tot), D(V[k, c])))
            out[i, c] = float(acc)
    return out


def pin_decimal_bruteforce(o):
    shapes = [(1, 1, 1, 1), (2, 3, 4, 5), (5, 7, 3, 2), (8, 8, 8, 8), (3, 6, 8, 1)]
    for t, (nq, nk, dk, dv) in enumerate(shapes):
        r = _rng(100 + t)
        Q = _f32(r.normal(size=(nq, dk)) * 2.0)
        K = _f32(r.normal(size=(nk, dk)))
        V = _f32(r.normal(size=(nk, dv)))
        scale = 1.0 / math.sqrt(dk)
        ref = decimal_attention(Q, K, V, scale)
        got = o.attn(Q, K, V, scale)
        err = np.max(np.abs(got - ref)) / max(1e-300, np.max(np.abs(ref)))
        assert err <= 1e-13, (nq, nk, dk, dv, err)


# ----------------------------------------------------------------------------------------------
# 3. Invariants and closed forms
# ----------------------------------------------------------------------------------------------
def pin_row_sums(o):
    for t, (nq, nk, dk) in enumerate([(7, 13, 5), (16, 300, 64), (3, 1, 8)]):
        r = _rng(200 + t)
        Q = _f32(r.normal(size=(nq, dk)) * 3)
        K = _f32(r.normal(size=(nk, dk)))
        V = _f32(r.normal(size=(nk, 4)))
        w, _ = o.weights(Q, K, V, 1.0 / math.sqrt(dk))
        assert np.all(w >= 0.0)
        assert np.max(np.abs(w.sum(axis=1) - 1.0)) <= nk * 1e-15 + 1e-15


def pin_v_ones(o):
    r = _rng(300)
    Q = _f32(r.normal(size=(2, 3, 33, 16)) * 4)
    K = _f32(r.normal(size=(2, 3, 71, 16)))
    V = np.ones((2, 3, 71, 8), dtype=np.float32)
    out = o.attn(Q, K, V, 0.25)
    assert np.max(np.abs(out - 1.0)) <= 1e-14


def pin_q_zero_column_mean(o):
    r = _rng(301)
    K = _f32(r.normal(size=(1, 2, 50, 8)))
    V = _f32(r.normal(size=(1, 2, 50, 6)))
    Q = np.zeros((1, 2, 9, 8), dtype=np.float32)
    mean = V.astype(np.float64).mean(axis=2, keepdims=True)
    out = o.attn(Q, K, V, 0.3)
    assert np.max(np.abs(out - mean)) <= 1e-14
    # scale = 0 gives the same, for any Q.
    Q2 = _f32(r.normal(size=(1, 2, 9, 8)))
    out2 = o.attn(Q2, K, V, 0.0)
    assert np.max(np.abs(out2 - mean)) <= 1e-14


def pin_single_key(o):
    r = _rng(302)
    Q = _f32(r.normal(size=(2, 2, 5, 8)) * 10)
    K = _f32(r.normal(size=(2, 2, 1, 8)))
    V = _f32(r.normal(size=(2, 2, 1, 3)))
    out = o.attn(Q, K, V, 0.7)
    assert np.array_equal(out, np.broadcast_to(V.astype(np.float64), out.shape))


def pin_two_keys_logistic(o):
    """Two keys: O = V0 + sigmoid(s1 - s0) (V1 - V0), with s_k = scale <q, k_k>."""
    r = _rng(303)
    Q = _f32(r.normal(size=(11, 6)))
    K = _f32(r.normal(size=(2, 6)))
    V = _f32(r.normal(size=(2, 5)))
    scale = 0.9
    q64, k64, v64 = Q.astype(np.float64), K.astype(np.float64), V.astype(np.float64)
    d = scale * (q64 @ k64[1] - q64 @ k64[0])
    sig = 1.0 / (1.0 + np.exp(-d))
    ref = v64[0][None, :] + sig[:, None] * (v64[1] - v64[0])[None, :]
    out = o.attn(Q, K, V, scale)
    assert np.max(np.abs(out - ref)) <= 1e-14


def pin_convexity(o):
    r = _rng(304)
    Q = _f32(r.normal(size=(1, 1, 40, 12)) * 5)
    K = _f32(r.normal(size=(1, 1, 90, 12)))
    V = _f32(r.normal(size=(1, 1, 90, 7)))
    out = o.attn(Q, K, V, 1.0 / math.sqrt(12))[0, 0]
    lo = V[0, 0].min(axis=0).astype(np.float64)
    hi = V[0, 0].max(axis=0).astype(np.float64)
    assert np.all(out >= lo[None, :] - 1e-15) and np.all(out <= hi[None, :] + 1e-15)


def pin_key_permutation_and_row_locality(o):
    r = _rng(305)
    Q = _f32(r.normal(size=(2, 2, 20, 8)))
    K = _f32(r.normal(size=(2, 2, 37, 8)))
    V = _f32(r.normal(size=(2, 2, 37, 5)))
    base = o.attn(Q, K, V, 0.35)
    perm = r.permutation(37)
    permd = o.attn(Q, K[:, :, perm], V[:, :, perm], 0.35)
    assert np.max(np.abs(permd - base)) <= 1e-14
    # Output row i depends on query row i only (and heads are independent).
    Q2 = Q.copy()
    Q2[1, 0, 3] = _f32(r.normal(size=8))
    changed = o.attn(Q2, K, V, 0.35)
    mask = np.ones(base.shape[:3], dtype=bool)
    mask[1, 0, 3] = False
    assert np.array_equal(changed[mask], base[mask])
    assert not np.array_equal(changed[1, 0, 3], base[1, 0, 3])
    # Rows of a query matrix flipped upside down give the output flipped the same way.
    flipped = o.attn(Q[:, :, ::-1], K, V, 0.35)
    assert np.array_equal(flipped, base[:, :, ::-1])


def pin_head_independence(o):
    """Each (b,h) slice is its own 2-D problem (Remark in Section 4.2)."""
    r = _rng(306)
    Q = _f32(r.normal(size=(2, 3, 9, 8)))
    K = _f32(r.normal(size=(2, 3, 14, 8)))
    V = _f32(r.normal(size=(2, 3, 14, 4)))
    full = o.attn(Q, K, V, 0.5)
    for b in range(2):
        for h in range(3):
            one = o.attn(Q[b, h], K[b, h], V[b, h], 0.5)
            assert np.array_equal(one, full[b, h])


def pin_shift_invariance(o):
    """Adding a constant to a score row leaves the output unchanged (Eq. stable_softmax)."""
    r = _rng(307)
    Q = _f32(r.normal(size=(1, 2, 10, 16)) * 2)
    K = _f32(r.normal(size=(1, 2, 33, 16)))
    V = _f32(r.normal(size=(1, 2, 33, 4)))
    base = o.attn(Q, K, V, 0.25)
    for c in (-1e3, 0.5, 1e3):
        sh = np.full(20, c)
        out = o.attn_shifted(Q, K, V, 0.25, sh)
        assert np.max(np.abs(out - base)) <= 1e-11, c
    # The same through the inputs: K[..,0] = 1 and Q[..,0] = delta adds scale*delta to row i.
    K2 = K.copy()
    K2[..., 0] = 1.0
    Qa = Q.copy()
    Qa[..., 0] = 0.0
    Qb = Qa.copy()
    Qb[..., 0] = _f32(r.integers(-64, 64, size=Qb.shape[:3]))
    a = o.attn(Qa, K2, V, 0.25)
    b = o.attn(Qb, K2, V, 0.25)
    assert np.max(np.abs(a - b)) <= 1e-12


def pin_large_scores_stable(o):
    """Scores of magnitude far beyond exp's range: max subtraction keeps them finite."""
    r = _rng(308)
    Q = _f32(r.normal(size=(1, 1, 6, 32)) * 40)
    K = _f32(r.normal(size=(1, 1, 25, 32)) * 40)
    V = _f32(r.normal(size=(1, 1, 25, 3)))
    s = o.scores(Q, K, 1.0)
    assert np.max(np.abs(s)) > 2000  # exp() of these would overflow without the shift
    out = o.attn(Q, K, V, 1.0)
    assert np.all(np.isfinite(out))
    # With such a spread, the softmax is one-hot on each row's arg-max key.
    top = np.argmax(s[0, 0], axis=1)
    srt = np.sort(s[0, 0], axis=1)
    assert np.all(srt[:, -1] - srt[:, -2] > 40)
    assert np.max(np.abs(out[0, 0] - V[0, 0][top].astype(np.float64))) <= 1e-15


def pin_planted_rows(o):
    """Q[i] := K[k*] with a margin > 30 over the next score gives O[i] = V[k*] (exp(-30) ~ 1e-13)."""
    r = _rng(309)
    K = _f32(r.normal(size=(1, 1, 64, 128)) * 8)
    V = _f32(r.normal(size=(1, 1, 64, 5)))
    Q = _f32(r.normal(size=(1, 1, 8, 128)) * 8)
    Q[0, 0, 3] = K[0, 0, 17]
    scale = 1.0 / math.sqrt(128)
    s = o.scores(Q, K, scale)[0, 0, 3]
    srt = np.sort(s)
    assert srt[-1] - srt[-2] > 30 and np.argmax(s) == 17
    out = o.attn(Q, K, V, scale)
    assert np.max(np.abs(out[0, 0, 3] - V[0, 0, 17])) <= 1e-12


def pin_rows_and_threads(o):
    """Sampled rows equal the full computation, and thread count does not change any bit."""
    r = _rng(310)
    Q = _f32(r.normal(size=(2, 2, 30, 16)))
    K = _f32(r.normal(size=(2, 2, 45, 16)))
    V = _f32(r.normal(size=(2, 2, 45, 8)))
    full1 = o.attn(Q, K, V, 0.25, nthreads=1)
    full4 = o.attn(Q, K, V, 0.25, nthreads=4)
    assert np.array_equal(full1, full4)
    rows = np.array([0, 29, 30, 77, 119])
    got = o.rows(Q, K, V, 0.25, rows)
    assert np.array_equal(got, full1.reshape(-1, 8)[rows])


def pin_lse(o):
    """Log-sum-exp of the scaled scores: decimal brute force, one key, and shift behaviour."""
    ctx = decimal.Context(prec=50)
    r = _rng(311)
    Q = _f32(r.normal(size=(4, 5)) * 3)
    K = _f32(r.normal(size=(6, 5)))
    V = _f32(r.normal(size=(6, 2)))
    _, lse = o.attn_lse(Q, K, V, 0.6)
    for i in range(4):
        tot = decimal.Decimal(0)
        for kk in range(6):
            s = decimal.Decimal(0)
            for j in range(5):
                s = ctx.add(s, ctx.multiply(decimal.Decimal(float(Q[i, j])), decimal.Decimal(float(K[kk, j]))))
            tot = ctx.add(tot, ctx.exp(ctx.multiply(s, decimal.Decimal(0.6))))
        assert abs(lse[i] - float(ctx.ln(tot))) <= 1e-13 * max(1.0, abs(lse[i]))
    # one key: lse = its scaled score; V plays no part
    K1 = K[:1]
    _, l1 = o.attn_lse(Q, K1, V[:1], 0.6)
    assert np.max(np.abs(l1 - 0.6 * (Q.astype(np.float64) @ K1[0].astype(np.float64)))) <= 1e-12
    _, l2 = o.attn_lse(Q, K, V * 3 + 1, 0.6)
    assert np.array_equal(lse, l2)
    # K[..,0] = 1, Q[..,0] = delta: every score of row i moves by scale*delta, lse too
    Ka = K.copy()
    Ka[:, 0] = 1.0
    Qa = Q.copy()
    Qa[:, 0] = 0.0
    Qb = Qa.copy()
    Qb[:, 0] = _f32([1.0, -2.0, 4.0, 8.0])
    _, la = o.attn_lse(Qa, Ka, V, 0.5)
    _, lb = o.attn_lse(Qb, Ka, V, 0.5)
    assert np.max(np.abs((lb - la) - 0.5 * np.array([1.0, -2.0, 4.0, 8.0]))) <= 1e-12


# ----------------------------------------------------------------------------------------------
# 4. Backward pass (Stage 5): gradients of L = sum(dO * O)
# ----------------------------------------------------------------------------------------------
def _decimal_loss(Q, K, V, G, scale, ctx):
    """L = sum_ic G[i,c] * O[i,c] with O = softmax(scale Q K^T) V, all in decimal arithmetic;
    Q, K, V, G are nested lists of Decimals."""
    nq, nk, dk, dv = len(Q), len(K), len(Q[0]), len(V[0])
    total = decimal.Decimal(0)
    for i in range(nq):
        ex = []
        for k in range(nk):
            s = decimal.Decimal(0)
            for j in range(dk):
                s = ctx.add(s, ctx.multiply(Q[i][j], K[k][j]))
            ex.append(ctx.exp(ctx.multiply(s, scale)))
        z = decimal.Decimal(0)
        for e in ex:
            z = ctx.add(z, e)
        for c in range(dv):
            acc = decimal.Decimal(0)
            for k in range(nk):
                acc = ctx.add(acc, ctx.multiply(ex[k], V[k][c]))
            total = ctx.add(total, ctx.multiply(G[i][c], ctx.divide(acc, z)))
    return total


def pin_bwd_finite_differences(o):
    """Every gradient entry against a central difference of the loss in 60-digit decimal
    arithmetic (step 1e-12: truncation ~1e-24, rounding ~1e-48)."""
    ctx = decimal.Context(prec=60)
    D = lambda x: decimal.Decimal(float(x))
    for t, (nq, nk, dk, dv, scale) in enumerate([(3, 4, 3, 2, 0.7), (2, 5, 2, 3, -1.3)]):
        r = _rng(400 + t)
        Q = _f32(r.normal(size=(nq, dk)) * 1.5)
        K = _f32(r.normal(size=(nk, dk)))
        V = _f32(r.normal(size=(nk, dv)))
        G = _f32(r.normal(size=(nq, dv)))
        dq, dkk, dvv = o.attn_bwd(Q, K, V, G, scale)
        mats = [[[D(x) for x in row] for row in M] for M in (Q, K, V)]
        g = [[D(x) for x in row] for row in G]
        sc = D(scale)
        h = decimal.Decimal("1e-12")
        for which, grad in enumerate((dq, dkk, dvv)):
            M = mats[which]
            for a in range(len(M)):
                for b in range(len(M[0])):
                    keep = M[a][b]
                    M[a][b] = keep + h
                    lp = _decimal_loss(mats[0], mats[1], mats[2], g, sc, ctx)
                    M[a][b] = keep - h
                    lm = _decimal_loss(mats[0], mats[1], mats[2], g, sc, ctx)
                    M[a][b] = keep
                    fd = float(ctx.divide(ctx.subtract(lp, lm), 2 * h))
                    assert abs(grad[a, b] - fd) <= 1e-12 * max(1.0, abs(fd)), (t, which, a, b)


def pin_bwd_closed_forms(o):
    """One key: dQ = dK = 0 and dV = sum_i dO_i.  scale = 0: dQ = dK = 0 and dV_k = mean
    over keys of sum_i dO_i.  Identical value rows: dQ = dK = 0."""
    r = _rng(410)
    Q = _f32(r.normal(size=(2, 3, 7, 8)) * 3)
    K = _f32(r.normal(size=(2, 3, 1, 8)))
    V = _f32(r.normal(size=(2, 3, 1, 5)))
    G = _f32(r.normal(size=(2, 3, 7, 5)))
    dq, dkk, dvv = o.attn_bwd(Q, K, V, G, 0.8)
    assert np.max(np.abs(dq)) == 0.0 and np.max(np.abs(dkk)) == 0.0
    assert np.max(np.abs(dvv[:, :, 0] - G.astype(np.float64).sum(axis=2))) <= 1e-13
    K = _f32(r.normal(size=(2, 3, 9, 8)))
    V = _f32(r.normal(size=(2, 3, 9, 5)))
    dq, dkk, dvv = o.attn_bwd(Q, K, V, G, 0.0)
    assert np.max(np.abs(dq)) == 0.0 and np.max(np.abs(dkk)) == 0.0
    mean = G.astype(np.float64).sum(axis=2, keepdims=True) / 9.0
    assert np.max(np.abs(dvv - mean)) <= 1e-13
    Vs = np.broadcast_to(V[:, :, :1], V.shape).copy()
    dq, dkk, _ = o.attn_bwd(Q, K, Vs, G, 0.5)
    assert np.max(np.abs(dq)) <= 1e-13 and np.max(np.abs(dkk)) <= 1e-13


def pin_bwd_invariants(o):
    """Each row of dS sums to zero, so the dK rows of a head sum to zero; the weights of a row
    sum to one, so the dV rows of a head sum to sum_i dO_i; by homogeneity of the scores in
    Q and in K, <dQ, Q> = <dK, K> per head; and the gradients are linear in dO."""
    r = _rng(411)
    Q = _f32(r.normal(size=(2, 2, 13, 16)) * 2)
    K = _f32(r.normal(size=(2, 2, 21, 16)))
    V = _f32(r.normal(size=(2, 2, 21, 6)))
    # dO values on a 1/64 grid, so that G1 + G2 is exact in float32
    G1 = _f32(np.round(r.normal(size=(2, 2, 13, 6)) * 64) / 64)
    G2 = _f32(np.round(r.normal(size=(2, 2, 13, 6)) * 64) / 64)
    dq, dkk, dvv = o.attn_bwd(Q, K, V, G1, 0.3)
    assert np.max(np.abs(dkk.sum(axis=2))) <= 1e-12 * np.max(np.abs(dkk))
    assert np.max(np.abs(dvv.sum(axis=2) - G1.astype(np.float64).sum(axis=2))) <= 1e-12
    qq = np.einsum("bhij,bhij->bh", dq, Q.astype(np.float64))
    kk = np.einsum("bhkj,bhkj->bh", dkk, K.astype(np.float64))
    assert np.max(np.abs(qq - kk)) <= 1e-12 * np.max(np.abs(qq))
    a = o.attn_bwd(Q, K, V, G1, 0.3)
    b = o.attn_bwd(Q, K, V, G2, 0.3)
    c = o.attn_bwd(Q, K, V, G1.astype(np.float64) + G2.astype(np.float64), 0.3)
    for x, y, z in zip(a, b, c):
        assert np.max(np.abs(x + y - z)) <= 1e-12 * max(1.0, np.max(np.abs(z)))
    # thread count does not change any bit
    assert all(np.array_equal(x, y) for x, y in zip(o.attn_bwd(Q, K, V, G1, 0.3, nthreads=1),
                                                    o.attn_bwd(Q, K, V, G1, 0.3, nthreads=3)))


# ----------------------------------------------------------------------------------------------
# 5. Input projections (Section 4.1): Q = X W_Q, K = X W_K, V = X W_V, stored head-major
# ----------------------------------------------------------------------------------------------
def pin_qkv_proj_exact_integers(o):
    """Small-integer X and W: every product and sum is exact, so the oracle must equal an
    integer brute force (Python ints) in the documented head-major layout."""
    r = _rng(500)
    B, N, d, H, dk, dv = 2, 5, 6, 3, 2, 4
    X = r.integers(-4, 5, size=(B, N, d))
    W = r.integers(-4, 5, size=(d, 2 * H * dk + H * dv))
    q, k, v = o.qkv_proj(_f32(X), _f32(W), H, dk, dv)
    for b in range(B):
        for n in range(N):
            for h in range(H):
                for j in range(dk):
                    eq = sum(int(X[b, n, c]) * int(W[c, h * dk + j]) for c in range(d))
                    ek = sum(int(X[b, n, c]) * int(W[c, H * dk + h * dk + j]) for c in range(d))
                    assert q[b, h, n, j] == eq and k[b, h, n, j] == ek
                for j in range(dv):
                    ev = sum(int(X[b, n, c]) * int(W[c, 2 * H * dk + h * dv + j]) for c in range(d))
                    assert v[b, h, n, j] == ev


def pin_qkv_proj_unit_columns(o):
    """W with one 1 per output column selects an input feature: the output must be that
    feature of X, at the head and position the column names (catches layout mix-ups)."""
    r = _rng(501)
    B, N, d, H, dk, dv = 2, 7, 9, 2, 3, 2
    X = _f32(r.normal(size=(B, N, d)))
    ncol = 2 * H * dk + H * dv
    src = r.integers(0, d, size=ncol)
    W = np.zeros((d, ncol), dtype=np.float32)
    W[src, np.arange(ncol)] = 1.0
    q, k, v = o.qkv_proj(X, W, H, dk, dv)
    for h in range(H):
        for j in range(dk):
            assert np.array_equal(q[:, h, :, j], X[:, :, src[h * dk + j]])
            assert np.array_equal(k[:, h, :, j], X[:, :, src[H * dk + h * dk + j]])
        for j in range(dv):
            assert np.array_equal(v[:, h, :, j], X[:, :, src[2 * H * dk + h * dv + j]])


ALL_PINS = [
    pin_paper_example,
    pin_decimal_bruteforce,
    pin_row_sums,
    pin_v_ones,
    pin_q_zero_column_mean,
    pin_single_key,
    pin_two_keys_logistic,
    pin_convexity,
    pin_key_permutation_and_row_locality,
    pin_head_independence,
    pin_shift_invariance,
    pin_large_scores_stable,
    pin_planted_rows,
    pin_rows_and_threads,
    pin_lse,
    pin_bwd_finite_differences,
    pin_bwd_closed_forms,
    pin_bwd_invariants,
    pin_qkv_proj_exact_integers,
    pin_qkv_proj_unit_columns,
]
