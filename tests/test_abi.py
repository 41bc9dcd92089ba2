"""The C ABI without a GPU: the library loads, exports every declared symbol, and rejects bad
arguments with the documented status codes before launching anything."""
import math
import os
import re

import numpy as np
import pytest

import paper_2606_07713_gb300 as pkg
from paper_2606_07713_gb300 import _lib
from paper_2606_07713_gb300 import inputs as I

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "moa_attn.h")


@pytest.fixture(scope="module")
def L():
    from paper_2606_07713_gb300 import build
    build.build()
    return _lib.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(moa_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    assert "moa_attn_fwd" in names and "moa_get_device_status" in names
    assert set(names) == set(_lib.SIGNATURES), "binding and header disagree"


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name
    assert pkg.moa_attn_version() >= 100


def test_flops_and_dnf_bytes_helpers(L):
    for cid, cfg in I.CONFIGS.items():
        s = cfg.shape
        f = pkg.attn_flops(s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v)
        assert f == 2.0 * s.B * s.H * s.N_q * s.N_k * (s.d_k + s.d_v)
        elt = 4 if cfg.dtype == "fp32" else 2
        code = pkg.MOA_FP32 if cfg.dtype == "fp32" else pkg.MOA_BF16
        b = pkg.dnf_bytes(s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v, code)
        assert b == elt * (s.numel_q + s.numel_k + s.numel_v + s.numel_o)
    assert math.isclose(pkg.attn_flops(2, 32, 8192, 8192, 128, 128), 2.199023e12, rel_tol=1e-6)
    assert pkg.dnf_bytes(1, 1, 1, 1, 1, 1, 9) == -1.0


# Fake, never dereferenced device addresses: validation fails before any CUDA call.
A, B_, C, D = 0x100000, 0x200000, 0x300000, 0x400000


def call(Q=A, K=B_, V=C, O=D, B=1, H=1, Nq=8, Nk=8, dk=64, dv=64, scale=0.125, dtype=1):
    return _lib.moa_attn_fwd(Q, K, V, O, B, H, Nq, Nk, dk, dv, scale, dtype, None)


@pytest.mark.parametrize("kwargs,code", [
    (dict(Q=None), _lib.MOA_ERR_INVALID_ARG),
    (dict(O=None), _lib.MOA_ERR_INVALID_ARG),
    (dict(B=0), _lib.MOA_ERR_INVALID_ARG),
    (dict(Nk=0), _lib.MOA_ERR_INVALID_ARG),
    (dict(dv=-1), _lib.MOA_ERR_INVALID_ARG),
    (dict(scale=float("nan")), _lib.MOA_ERR_INVALID_ARG),
    (dict(scale=float("inf")), _lib.MOA_ERR_INVALID_ARG),
    (dict(dtype=7), _lib.MOA_ERR_UNSUPPORTED_DTYPE),
    (dict(dk=96), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
    (dict(dv=256), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
    (dict(dtype=0, dk=132), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
    (dict(dtype=0, dv=6), _lib.MOA_ERR_MISALIGNED),
    (dict(Q=A + 8), _lib.MOA_ERR_MISALIGNED),
    (dict(O=D + 2), _lib.MOA_ERR_MISALIGNED),
    (dict(O=A), _lib.MOA_ERR_INVALID_ARG),              # O aliases Q
    (dict(O=C + 16), _lib.MOA_ERR_INVALID_ARG),         # O overlaps V
    (dict(Nq=2 ** 31), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
    (dict(B=2 ** 20, H=2 ** 12), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
    (dict(B=2 ** 40, Nq=2 ** 20), _lib.MOA_ERR_UNSUPPORTED_SHAPE),
])
def test_validation_rejects_before_launch(L, kwargs, code):
    assert call(**kwargs) == code
    assert _lib.moa_last_error() != ""


def test_staged_rejects_null_host_pointers(L):
    rc = _lib.moa_attn_fwd_staged(None, A, A, A, A, B_, C, D, 1, 1, 8, 8, 64, 64, 0.1, 1, None)
    assert rc == _lib.MOA_ERR_INVALID_ARG


def test_splitkv_workspace_formula(L):
    ws = pkg.moa_attn_splitkv_workspace_bytes
    # 1000 keys = 8 blocks; 3 splits of 3,3,2 blocks
    assert ws(1, 2, 256, 1000, 64, 64, pkg.MOA_BF16, 3) == 3 * 2 * 256 * (4 * 64 + 8)
    # more splits than blocks: one split per block
    assert ws(1, 1, 10, 300, 64, 128, pkg.MOA_BF16, 9) == 3 * 10 * (4 * 128 + 8)
    # 8 blocks in 5 requested splits: 2 blocks each -> 4 splits
    assert ws(1, 1, 10, 1024, 64, 64, pkg.MOA_BF16, 5) == 4 * 10 * (4 * 64 + 8)
    assert ws(1, 1, 10, 128, 64, 64, pkg.MOA_BF16, 4) == 0      # one block: no split
    assert ws(1, 1, 10, 1024, 64, 64, pkg.MOA_FP32, 4) == 0     # fp32 has no split form
    assert ws(0, 1, 10, 1024, 64, 64, pkg.MOA_BF16, 4) == 0


def test_splitkv_validation_without_gpu(L):
    f = _lib.moa_attn_fwd_splitkv
    assert f(A, B_, C, D, 1, 1, 8, 1024, 64, 64, 0.1, 1, -1, 0x500000, 1 << 20, None) == _lib.MOA_ERR_INVALID_ARG
    assert f(A, B_, C, D, 1, 1, 8, 1024, 64, 64, 0.1, 1, 4, None, 0, None) == _lib.MOA_ERR_INVALID_ARG
    assert f(A, B_, C, D, 1, 1, 8, 1024, 64, 64, 0.1, 1, 4, 0x500008, 1 << 20, None) == _lib.MOA_ERR_MISALIGNED
    assert f(A, B_, C, D, 1, 1, 8, 1024, 64, 64, 0.1, 1, 4, D, 1 << 20, None) == _lib.MOA_ERR_INVALID_ARG


def test_split_plan_of_the_workloads(L):
    """The library's own split on a 152-SM GPU: only shapes whose query blocks leave SMs idle."""
    plan = pkg.moa_attn_split_plan
    auto = pkg.MOA_SPLITS_AUTO
    # a wave or more of query blocks: nothing is split (the plain kernel runs)
    assert plan(4, 16, 2048, 2048, auto, 152) == (0, 1, 16, 512)
    assert plan(2, 32, 8192, 8192, auto, 152) == (0, 1, 64, 2048)
    assert plan(8, 8, 1024, 4096, auto, 152) == (0, 1, 32, 256)
    assert plan(1, 152, 256, 4096, auto, 152) == (0, 1, 32, 152)
    # 16 blocks, 256 key blocks: 9 splits of 29 blocks fill 144 SMs in one round
    assert plan(1, 16, 256, 32768, auto, 152) == (0, 9, 29, 0)
    # 8 blocks, 512 key blocks: 16 splits of 32 blocks (at most 32 splits; 19 would not
    # save 2 % more)
    assert plan(1, 8, 128, 65536, auto, 152) == (0, 16, 32, 0)
    # 100 blocks of 16 key blocks: any split needs two rounds; not worth it
    assert plan(1, 100, 256, 2048, auto, 152) == (0, 1, 16, 100)
    # too few key blocks to split (each range keeps two)
    assert plan(1, 2, 256, 300, auto, 152) == (0, 1, 3, 2)
    # a requested count splits every block
    assert plan(1, 2, 256, 1000, 3, 152) == (0, 3, 3, 0)
    assert plan(1, 2, 256, 1000, 1, 152) == (0, 1, 8, 2)
    assert plan(1, 2, 256, 1000, -1, 152)[0] == _lib.MOA_ERR_INVALID_ARG
    assert plan(0, 2, 256, 1000, auto, 152)[0] == _lib.MOA_ERR_INVALID_ARG
    assert plan(1, 2, 256, -5, auto, 152)[0] == _lib.MOA_ERR_INVALID_ARG


def test_split_plan_properties(L):
    """Over random shapes and SM counts, the automatic plan is well formed: it splits only
    when the query blocks fill less than one wave, every key range is non-empty with at
    least two key blocks, and the split CTAs are predicted to take at most 0.85 of the time."""
    rng = np.random.default_rng(7)
    n_split = 0
    for _ in range(3000):
        B, H = int(rng.integers(1, 5)), int(rng.integers(1, 33))
        Nq, Nk = int(rng.integers(1, 4000)), int(rng.integers(1, 70000))
        sms = int(rng.integers(1, 300))
        rc, s, per, whole = pkg.moa_attn_split_plan(B, H, Nq, Nk, pkg.MOA_SPLITS_AUTO, sms)
        assert rc == 0
        units = B * H * -(-Nq // 256)
        n_kt = -(-Nk // 128)
        if s == 1:
            assert whole == units and per == n_kt
            continue
        n_split += 1
        assert units < sms and whole == 0
        assert per >= 2 and (s - 1) * per < n_kt <= s * per and s <= 32
        rounds = -(-(units * s) // sms)
        assert rounds * (per / n_kt + 0.08) <= 0.85 + 1e-9
    assert n_split > 100


def test_lse_validation_without_gpu(L):
    f = _lib.moa_attn_fwd_lse
    E = 0x500000
    ok_args = (1, 1, 8, 8, 64, 64, 0.125, 1, None)
    assert f(A, B_, C, D, None, *ok_args) == _lib.MOA_ERR_INVALID_ARG        # no LSE buffer
    assert f(A, B_, C, D, E + 2, *ok_args) == _lib.MOA_ERR_MISALIGNED        # not 4-byte aligned
    assert f(A, B_, C, D, D + 4, *ok_args) == _lib.MOA_ERR_INVALID_ARG       # LSE inside O
    assert f(A, B_, C, D, A, *ok_args) == _lib.MOA_ERR_INVALID_ARG           # LSE aliases Q
    assert f(None, B_, C, D, E, *ok_args) == _lib.MOA_ERR_INVALID_ARG        # the usual checks too
    assert f(A, B_, C, D, E, 1, 1, 8, 8, 96, 64, 0.125, 1, None) == _lib.MOA_ERR_UNSUPPORTED_SHAPE


def test_bwd_fused_workspace_formula_and_validation(L):
    ws = pkg.moa_attn_bwd_fused_workspace_bytes
    assert ws(2, 3, 200, 300, 64, 64, pkg.MOA_BF16) == 2 * 3 * 256 * 4 * (2 + 64)
    assert ws(1, 1, 128, 5, 64, 64, pkg.MOA_BF16) == 128 * 4 * 66
    assert ws(1, 1, 128, 5, 128, 64, pkg.MOA_BF16) == 0     # d_k = d_v = 64 only
    assert ws(1, 1, 128, 5, 64, 64, pkg.MOA_FP32) == 0
    assert ws(0, 1, 128, 5, 64, 64, pkg.MOA_BF16) == 0
    f = _lib.moa_attn_bwd_fused
    E = 0x600000
    args = (1, 1, 128, 128, 64, 64, 0.125, 1)
    W = 0x700000
    need = ws(1, 1, 128, 128, 64, 64, pkg.MOA_BF16)
    # workspace too small, misaligned, overlapping; other head sizes; fp32
    assert f(A, B_, C, D, E, 0x680000, 0x800000, 0x810000, 0x820000, *args, W, need - 16, None) == _lib.MOA_ERR_INVALID_ARG
    assert f(A, B_, C, D, E, 0x680000, 0x800000, 0x810000, 0x820000, *args, W + 8, need, None) == _lib.MOA_ERR_MISALIGNED
    assert f(A, B_, C, D, E, 0x680000, 0x800000, 0x810000, 0x820000, *args, A, need, None) == _lib.MOA_ERR_INVALID_ARG
    assert f(A, B_, C, D, E, 0x680000, 0x800000, 0x810000, 0x820000, 1, 1, 128, 128, 128, 128, 0.125, 1, W, 1 << 24, None) == _lib.MOA_ERR_UNSUPPORTED_SHAPE
    assert f(A, B_, C, D, E, 0x680000, 0x800000, 0x810000, 0x820000, 1, 1, 128, 128, 64, 64, 0.125, 0, W, 1 << 24, None) == _lib.MOA_ERR_UNSUPPORTED_DTYPE


def test_bwd_workspace_formula(L):
    ws = pkg.moa_attn_bwd_workspace_bytes
    assert ws(2, 3, 200, 300, 64, 64, pkg.MOA_BF16) == 2 * 2 * 3 * 256 * 4
    assert ws(1, 1, 128, 5, 128, 64, pkg.MOA_BF16) == 2 * 128 * 4
    assert ws(1, 1, 128, 5, 128, 64, pkg.MOA_FP32) == 2 * 128 * 4      # same layout for fp32
    assert ws(1, 1, 128, 5, 128, 64, 7) == 0
    assert ws(0, 1, 128, 5, 128, 64, pkg.MOA_BF16) == 0


def test_bwd_validation_without_gpu(L):
    f = _lib.moa_attn_bwd
    # Q, K, V, O, dO, LSE, dQ, dK, dV, workspace: fake addresses 1 MiB apart
    P = [0x1000000 * (i + 1) for i in range(10)]
    dims = (1, 1, 8, 8, 64, 64, 0.125)

    def call(ptrs=None, dtype=1, ws_bytes=1 << 20, d=dims):
        p = list(P if ptrs is None else ptrs)
        return f(*p[:9], *d, dtype, p[9], ws_bytes, None)

    for i in range(4, 9):  # null dO, LSE or an output
        q = list(P)
        q[i] = None
        assert call(q) == _lib.MOA_ERR_INVALID_ARG
    assert call(dtype=7) == _lib.MOA_ERR_UNSUPPORTED_DTYPE
    assert call(d=(1, 1, 8, 8, 96, 64, 0.125)) == _lib.MOA_ERR_UNSUPPORTED_SHAPE
    assert call(dtype=0, d=(1, 1, 8, 8, 132, 64, 0.125)) == _lib.MOA_ERR_UNSUPPORTED_SHAPE
    assert call(ws_bytes=100) == _lib.MOA_ERR_INVALID_ARG               # workspace too small
    q = list(P); q[9] = None
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                          # no workspace
    q = list(P); q[6] = P[6] + 8
    assert call(q) == _lib.MOA_ERR_MISALIGNED                           # dQ misaligned
    q = list(P); q[5] = P[5] + 2
    assert call(q) == _lib.MOA_ERR_MISALIGNED                           # LSE misaligned
    q = list(P); q[7] = P[0]
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                          # dK aliases Q
    q = list(P); q[8] = P[6]
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                          # dV aliases dQ
    q = list(P); q[9] = P[4]
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                          # workspace aliases dO


def test_qkv_proj_validation_without_gpu(L):
    f = _lib.moa_qkv_proj
    P = [0x1000000 * (i + 1) for i in range(5)]   # X, W, Q, K, V
    ok = (2, 256, 512, 4, 64, 64)

    def call(p=None, dims=ok, dtype=1):
        return f(*(P if p is None else p), *dims, dtype, None)

    for i in range(5):
        q = list(P); q[i] = None
        assert call(q) == _lib.MOA_ERR_INVALID_ARG
    assert call(dtype=0) == _lib.MOA_ERR_UNSUPPORTED_DTYPE
    assert call(dims=(2, 256, 512, 4, 96, 64)) == _lib.MOA_ERR_UNSUPPORTED_SHAPE
    assert call(dims=(2, 256, 500, 4, 64, 64)) == _lib.MOA_ERR_MISALIGNED   # d_model % 8
    assert call(dims=(0, 256, 512, 4, 64, 64)) == _lib.MOA_ERR_INVALID_ARG
    q = list(P); q[3] = P[3] + 8
    assert call(q) == _lib.MOA_ERR_MISALIGNED
    q = list(P); q[2] = P[0]
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                            # Q aliases X
    q = list(P); q[4] = P[3] + 64
    assert call(q) == _lib.MOA_ERR_INVALID_ARG                            # V inside K
