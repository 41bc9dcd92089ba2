"""fp64 CPU oracle for scaled dot-product attention (ctypes wrapper).

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the CPU
baseline leg of bench.py may import this package.  The CUDA library never calls
it and has no fallback to it.

The arithmetic lives in attn_oracle.c (plain C, fp64, one row at a time in the
order of the paper's Algorithm 1).  This file only builds that library with
gcc, loads it and converts numpy arrays.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attn_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

CFLAGS = ["-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
          "-ffp-contract=off", "-Wall", "-Wextra"]


def build(force: bool = False) -> str:
    """Compile attn_oracle.c into oracle/_build/liboracle.so (gcc, OpenMP)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", *CFLAGS, _SRC, "-o", tmp, "-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError("oracle build failed:\n" + " ".join(cmd) + "\n" + r.stderr)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load(path: str | None = None):
    global _lib
    if path is None and _lib is not None:
        return _lib
    with _lock:
        if path is None and _lib is not None:
            return _lib
        lib = ctypes.CDLL(path or build())
        f64p = ctypes.POINTER(ctypes.c_double)
        f32p = ctypes.POINTER(ctypes.c_float)
        i64 = ctypes.c_int64
        i64p = ctypes.POINTER(ctypes.c_int64)
        lib.moa_oracle_attn_f64.argtypes = [f32p, f32p, f32p, f64p, i64, i64, i64, i64, i64, i64,
                                            ctypes.c_double, ctypes.c_int]
        lib.moa_oracle_rows_f64.argtypes = [f32p, f32p, f32p, f64p, i64, i64, i64, i64, i64, i64,
                                            ctypes.c_double, i64p, i64, ctypes.c_int]
        lib.moa_oracle_weights_f64.argtypes = [f32p, f32p, f32p, f64p, f64p, i64, i64, i64, i64,
                                               i64, i64, ctypes.c_double, ctypes.c_int]
        lib.moa_oracle_scores_f64.argtypes = [f32p, f32p, i64, i64, i64, i64, i64,
                                              ctypes.c_double, f64p, ctypes.c_int]
        lib.moa_oracle_attn_shifted_f64.argtypes = [f32p, f32p, f32p, f64p, i64, i64, i64, i64,
                                                    i64, i64, ctypes.c_double, f64p, ctypes.c_int]
        lib.moa_oracle_attn_lse_f64.argtypes = [f32p, f32p, f32p, f64p, f64p, i64, i64, i64,
                                                i64, i64, i64, ctypes.c_double, ctypes.c_int]
        lib.moa_oracle_attn_bwd_f64.argtypes = [f32p, f32p, f32p, f32p, f64p, f64p, f64p, i64,
                                                i64, i64, i64, i64, i64, ctypes.c_double,
                                                ctypes.c_int]
        lib.moa_oracle_qkv_proj_f64.argtypes = [f32p, f32p, f64p, f64p, f64p, i64, i64, i64, i64,
                                                i64, i64, ctypes.c_int]
        for name in ("moa_oracle_qkv_proj_f64", "moa_oracle_attn_bwd_f64", "moa_oracle_attn_lse_f64", "moa_oracle_attn_f64", "moa_oracle_rows_f64", "moa_oracle_weights_f64",
                     "moa_oracle_scores_f64", "moa_oracle_attn_shifted_f64",
                     "moa_oracle_max_threads"):
            getattr(lib, name).restype = ctypes.c_int
        if path is None:
            _lib = lib
        return lib


class Oracle:
    """numpy front end over one loaded copy of the oracle library."""

    def __init__(self, lib_path: str | None = None):
        self.lib = _load(lib_path)

    # -- helpers -------------------------------------------------------------------------
    @staticmethod
    def _f32(x):
        a = np.ascontiguousarray(x, dtype=np.float32)
        return a, a.ctypes.data_as(ctypes.POINTER(ctypes.c_float))

    @staticmethod
    def _dims(q, k, v):
        if q.ndim == 2:
            q, k, v = q[None, None], k[None, None], v[None, None]
        B, H, Nq, dk = q.shape
        Bk, Hk, Nk, dk2 = k.shape
        Bv, Hv, Nk2, dv = v.shape
        if (B, H) != (Bk, Hk) or (B, H) != (Bv, Hv) or dk != dk2 or Nk != Nk2:
            raise ValueError(f"inconsistent shapes {q.shape} {k.shape} {v.shape}")
        return q, k, v, (B, H, Nq, Nk, dk, dv)

    @staticmethod
    def _check(rc, what):
        if rc != 0:
            raise RuntimeError(f"{what} failed with status {rc}")

    # -- entry points --------------------------------------------------------------------
    def attn(self, q, k, v, scale: float, nthreads: int = 0) -> np.ndarray:
        """O = softmax(scale * Q K^T) V in fp64; q/k/v are [B,H,N,d] or [N,d]."""
        squeeze = np.ndim(q) == 2
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        out = np.empty((B, H, Nq, dv), dtype=np.float64)
        rc = self.lib.moa_oracle_attn_f64(qp, kp, vp, out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                                          B, H, Nq, Nk, dk, dv, float(scale), int(nthreads))
        self._check(rc, "moa_oracle_attn_f64")
        return out[0, 0] if squeeze else out

    def rows(self, q, k, v, scale: float, rows, nthreads: int = 0) -> np.ndarray:
        """Output rows for flattened row indices r = (b*H + h)*N_q + i; shape [len(rows), d_v]."""
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        r = np.ascontiguousarray(rows, dtype=np.int64)
        out = np.empty((r.size, dv), dtype=np.float64)
        rc = self.lib.moa_oracle_rows_f64(qp, kp, vp, out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                                          B, H, Nq, Nk, dk, dv, float(scale),
                                          r.ctypes.data_as(ctypes.POINTER(ctypes.c_int64)), r.size,
                                          int(nthreads))
        self._check(rc, "moa_oracle_rows_f64")
        return out

    def weights(self, q, k, v, scale: float, nthreads: int = 0):
        """(W, O): attention weights [B,H,N_q,N_k] and output [B,H,N_q,d_v]."""
        squeeze = np.ndim(q) == 2
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        w = np.empty((B, H, Nq, Nk), dtype=np.float64)
        o = np.empty((B, H, Nq, dv), dtype=np.float64)
        dp = ctypes.POINTER(ctypes.c_double)
        rc = self.lib.moa_oracle_weights_f64(qp, kp, vp, w.ctypes.data_as(dp), o.ctypes.data_as(dp),
                                             B, H, Nq, Nk, dk, dv, float(scale), int(nthreads))
        self._check(rc, "moa_oracle_weights_f64")
        return (w[0, 0], o[0, 0]) if squeeze else (w, o)

    def scores(self, q, k, scale: float, nthreads: int = 0) -> np.ndarray:
        """Scaled scores scale * Q K^T, [B,H,N_q,N_k]."""
        squeeze = np.ndim(q) == 2
        if squeeze:
            q, k = q[None, None], k[None, None]
        B, H, Nq, dk = q.shape
        Nk = k.shape[2]
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        s = np.empty((B, H, Nq, Nk), dtype=np.float64)
        rc = self.lib.moa_oracle_scores_f64(qp, kp, B, H, Nq, Nk, dk, float(scale),
                                            s.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                                            int(nthreads))
        self._check(rc, "moa_oracle_scores_f64")
        return s[0, 0] if squeeze else s

    def attn_shifted(self, q, k, v, scale: float, shift, nthreads: int = 0) -> np.ndarray:
        """Like attn() but with shift[r] added to every score of output row r."""
        squeeze = np.ndim(q) == 2
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        sh = np.ascontiguousarray(shift, dtype=np.float64).reshape(-1)
        if sh.size != B * H * Nq:
            raise ValueError("shift needs one value per output row")
        out = np.empty((B, H, Nq, dv), dtype=np.float64)
        dp = ctypes.POINTER(ctypes.c_double)
        rc = self.lib.moa_oracle_attn_shifted_f64(qp, kp, vp, out.ctypes.data_as(dp), B, H, Nq, Nk,
                                                  dk, dv, float(scale), sh.ctypes.data_as(dp),
                                                  int(nthreads))
        self._check(rc, "moa_oracle_attn_shifted_f64")
        return out[0, 0] if squeeze else out

    def attn_lse(self, q, k, v, scale: float, nthreads: int = 0):
        """(O, LSE): the output and, per output row, ln sum_k exp(scale * <q_i, k_k>)."""
        squeeze = np.ndim(q) == 2
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        out = np.empty((B, H, Nq, dv), dtype=np.float64)
        lse = np.empty((B, H, Nq), dtype=np.float64)
        dp = ctypes.POINTER(ctypes.c_double)
        rc = self.lib.moa_oracle_attn_lse_f64(qp, kp, vp, out.ctypes.data_as(dp),
                                              lse.ctypes.data_as(dp), B, H, Nq, Nk, dk, dv,
                                              float(scale), int(nthreads))
        self._check(rc, "moa_oracle_attn_lse_f64")
        return (out[0, 0], lse[0, 0]) if squeeze else (out, lse)

    def attn_bwd(self, q, k, v, do, scale: float, nthreads: int = 0):
        """(dQ, dK, dV) of L with dL/dO = do, for O = softmax(scale Q K^T) V, in fp64."""
        squeeze = np.ndim(q) == 2
        q, k, v, (B, H, Nq, Nk, dk, dv) = self._dims(q, k, v)
        if squeeze:
            do = np.asarray(do)[None, None]
        if tuple(np.shape(do)) != (B, H, Nq, dv):
            raise ValueError(f"dO must be {(B, H, Nq, dv)}, got {np.shape(do)}")
        q, qp = self._f32(q)
        k, kp = self._f32(k)
        v, vp = self._f32(v)
        g, gp = self._f32(do)
        dq = np.empty((B, H, Nq, dk), dtype=np.float64)
        dkk = np.empty((B, H, Nk, dk), dtype=np.float64)
        dvv = np.empty((B, H, Nk, dv), dtype=np.float64)
        dp = ctypes.POINTER(ctypes.c_double)
        rc = self.lib.moa_oracle_attn_bwd_f64(qp, kp, vp, gp, dq.ctypes.data_as(dp),
                                              dkk.ctypes.data_as(dp), dvv.ctypes.data_as(dp),
                                              B, H, Nq, Nk, dk, dv, float(scale), int(nthreads))
        self._check(rc, "moa_oracle_attn_bwd_f64")
        if squeeze:
            return dq[0, 0], dkk[0, 0], dvv[0, 0]
        return dq, dkk, dvv

    def qkv_proj(self, x, w, H: int, dk: int, dv: int, nthreads: int = 0):
        """(Q, K, V) = X W_Q, X W_K, X W_V in fp64, head-major [B, H, N, d]; x [B, N, d_model],
        w [d_model, 2*H*dk + H*dv] (W_Q | W_K | W_V)."""
        B, N, d = np.shape(x)
        if tuple(np.shape(w)) != (d, 2 * H * dk + H * dv):
            raise ValueError(f"w must be {(d, 2 * H * dk + H * dv)}, got {np.shape(w)}")
        x, xp = self._f32(x)
        w, wp = self._f32(w)
        q = np.empty((B, H, N, dk), dtype=np.float64)
        k = np.empty((B, H, N, dk), dtype=np.float64)
        v = np.empty((B, H, N, dv), dtype=np.float64)
        dp = ctypes.POINTER(ctypes.c_double)
        rc = self.lib.moa_oracle_qkv_proj_f64(xp, wp, q.ctypes.data_as(dp), k.ctypes.data_as(dp),
                                              v.ctypes.data_as(dp), B, N, d, H, dk, dv,
                                              int(nthreads))
        self._check(rc, "moa_oracle_qkv_proj_f64")
        return q, k, v

    def max_threads(self) -> int:
        return int(self.lib.moa_oracle_max_threads())


_default = None


def get() -> Oracle:
    """The oracle built from attn_oracle.c (built on first use)."""
    global _default
    if _default is None:
        _default = Oracle()
    return _default


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
