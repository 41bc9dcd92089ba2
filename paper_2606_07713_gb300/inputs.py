"""Seeded synthetic inputs for scaled dot-product attention.

This module is shared by the CUDA path (bench, tests) and by the CPU oracle's
tests.  It holds no attention arithmetic: it only draws numbers and rounds them
to the storage type.  Every value is a pure function of (seed, stream, index),
so the oracle and the kernels always see identical inputs.

Generator (all in float64, vectorised with numpy):

* splitmix64 (Steele, Lea, Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014) used counter-style: output i of stream (seed, s)
  is mix64(key + (i + 1) * 0x9E3779B97F4A7C15) with key = mix64(seed * 2^8 + s).
* 53-bit uniforms u = (z >> 11) * 2^-53, and u' = u + 2^-53 in (0, 1] where a
  logarithm is taken.
* Box-Muller (1958): a pair (u1', u2) gives r*cos(2 pi u2), r*sin(2 pi u2) with
  r = sqrt(-2 ln u1').
* Rounding: float64 -> float32 (round to nearest even), and for bf16 storage
  float32 -> bf16 by round-to-nearest-even on the bit pattern.

Streams: Q = 0, K = 1, V = 2, planted rows = 3.

Planted rows: per head, distinct query rows i_r and distinct keys k_r are drawn from stream 3,
and Q[i_r] is set to the stored K[k_r].  With a plant margin (the stability workload uses
PLANT_MARGIN), a drawn key is kept only if, in float64 on the stored values, the row's score for
k_r beats every other key's score by more than the margin (scores are scale * <q, k>);
otherwise the next key is drawn from the same stream.  This inner product is the input recipe's acceptance test, not an attention step: both
the oracle and the kernels receive the finished arrays.

The five workload shapes follow the paper's problem statement (Section 4.1,
Eq. attention, with the batched/multi-head layout of the Remark in Section 4.2):
Q [B,H,N_q,d_k], K [B,H,N_k,d_k], V [B,H,N_k,d_v], contiguous row-major.
"""
from __future__ import annotations

import concurrent.futures
import dataclasses
import math
import os
from typing import Optional

import numpy as np

_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)
_CHUNK = 1 << 20

STREAM_Q, STREAM_K, STREAM_V, STREAM_PLANT, STREAM_DO = 0, 1, 2, 3, 4

PLANT_MARGIN = 30.0     # a planted key's score must beat the row's next best by more than this
PLANT_MAX_DRAWS = 64    # key candidates drawn per planted row before the recipe gives up


def _mix64(z: np.ndarray) -> np.ndarray:
    z = (z ^ (z >> np.uint64(30))) * _M1
    z = (z ^ (z >> np.uint64(27))) * _M2
    return z ^ (z >> np.uint64(31))


def _stream_key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        base = np.array([(int(seed) << 8) + int(stream)], dtype=np.uint64)
        return _mix64(base)[0]


def raw_u64(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """Outputs start .. start+count-1 of the counter-based splitmix64 stream."""
    key = _stream_key(seed, stream)
    idx = np.arange(start + 1, start + count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        return _mix64(key + idx * _GOLDEN)


def uniform01(seed: int, stream: int, start: int, count: int) -> np.ndarray:
    """53-bit uniforms in [0, 1)."""
    z = raw_u64(seed, stream, start, count)
    return (z >> np.uint64(11)).astype(np.float64) * (2.0 ** -53)


def _pool_map(fn, jobs):
    """Run independent chunk jobs on a thread pool (numpy releases the GIL)."""
    if len(jobs) <= 1:
        for j in jobs:
            fn(*j)
        return
    workers = max(1, min(len(jobs), os.cpu_count() or 1, 32))
    with concurrent.futures.ThreadPoolExecutor(workers) as ex:
        list(ex.map(lambda j: fn(*j), jobs))


def normal(seed: int, stream: int, count: int) -> np.ndarray:
    """count i.i.d. N(0,1) draws in float64 (Box-Muller on consecutive pairs)."""
    out = np.empty(count, dtype=np.float64)
    npairs = (count + 1) // 2

    def chunk(p0, p1):
        u = uniform01(seed, stream, 2 * p0, 2 * (p1 - p0))
        u1 = u[0::2] + 2.0 ** -53          # (0, 1]: the logarithm stays finite
        u2 = u[1::2]
        r = np.sqrt(-2.0 * np.log(u1))
        t = (2.0 * math.pi) * u2
        pair = np.empty(2 * (p1 - p0), dtype=np.float64)
        pair[0::2] = r * np.cos(t)
        pair[1::2] = r * np.sin(t)
        lo = 2 * p0
        hi = min(count, 2 * p1)
        out[lo:hi] = pair[: hi - lo]

    _pool_map(chunk, [(p0, min(npairs, p0 + _CHUNK)) for p0 in range(0, npairs, _CHUNK)])
    return out


def uniform(seed: int, stream: int, count: int, lo: float, hi: float) -> np.ndarray:
    out = np.empty(count, dtype=np.float64)

    def chunk(c0, c1):
        out[c0:c1] = lo + (hi - lo) * uniform01(seed, stream, c0, c1 - c0)

    _pool_map(chunk, [(c0, min(count, c0 + _CHUNK)) for c0 in range(0, count, _CHUNK)])
    return out


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns the uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (b >> np.uint32(16)) & np.uint32(1)
    r = (b + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclasses.dataclass(frozen=True)
class AttnShape:
    B: int
    H: int
    N_q: int
    N_k: int
    d_k: int
    d_v: int

    @property
    def numel_q(self) -> int:
        return self.B * self.H * self.N_q * self.d_k

    @property
    def numel_k(self) -> int:
        return self.B * self.H * self.N_k * self.d_k

    @property
    def numel_v(self) -> int:
        return self.B * self.H * self.N_k * self.d_v

    @property
    def numel_o(self) -> int:
        return self.B * self.H * self.N_q * self.d_v


@dataclasses.dataclass(frozen=True)
class AttnConfig:
    """One synthetic workload: shape, storage type and value distributions."""
    cfg_id: int
    name: str
    shape: AttnShape
    dtype: str                 # "fp32" or "bf16"
    q_sigma: float = 1.0       # Q ~ q_sigma * N(0,1)
    k_sigma: float = 1.0       # K ~ k_sigma * N(0,1)
    v_dist: str = "normal"     # "normal" -> N(0,1); "uniform" -> U[-1,1]
    plants_per_head: int = 0   # rows i with Q[i] := K[k*]
    # planted key must beat the row's next best score by more than this (None: any key)
    plant_margin: Optional[float] = None
    seed: Optional[int] = None

    @property
    def scale(self) -> float:
        return 1.0 / math.sqrt(self.shape.d_k)

    @property
    def the_seed(self) -> int:
        return self.cfg_id if self.seed is None else self.seed


# The five workloads (shapes, dtypes, distributions); seed = workload number.
CONFIGS = {
    1: AttnConfig(1, "fp32 B1 H1 N128 d64", AttnShape(1, 1, 128, 128, 64, 64), "fp32"),
    2: AttnConfig(2, "bf16 B4 H16 N2048 d64", AttnShape(4, 16, 2048, 2048, 64, 64), "bf16"),
    3: AttnConfig(3, "bf16 B2 H32 N8192 d128", AttnShape(2, 32, 8192, 8192, 128, 128), "bf16"),
    4: AttnConfig(4, "bf16 B8 H8 Nq1024 Nk4096 dk128 dv64", AttnShape(8, 8, 1024, 4096, 128, 64),
                  "bf16", v_dist="uniform"),
    5: AttnConfig(5, "bf16 B1 H16 N32768 d128 stress (QK sigma 8, planted rows)",
                  AttnShape(1, 16, 32768, 32768, 128, 128), "bf16",
                  q_sigma=8.0, k_sigma=8.0, plants_per_head=8, plant_margin=PLANT_MARGIN),
}


@dataclasses.dataclass
class AttnInputs:
    """Inputs in the exact values the kernels see.

    q, k, v: float32 arrays [B,H,N,d] holding the stored values exactly (bf16
    values are exactly representable in float32).  For bf16 storage, q_bits,
    k_bits, v_bits hold the uint16 patterns.  plants: list of (b, h, i, k*).
    """
    cfg: AttnConfig
    q: np.ndarray
    k: np.ndarray
    v: np.ndarray
    q_bits: Optional[np.ndarray] = None
    k_bits: Optional[np.ndarray] = None
    v_bits: Optional[np.ndarray] = None
    plants: tuple = ()
    plant_redraws: int = 0     # key candidates rejected by the margin rule

    @property
    def shape(self) -> AttnShape:
        return self.cfg.shape

    @property
    def scale(self) -> float:
        return self.cfg.scale


def _store(x64: np.ndarray, dtype: str):
    x32 = x64.astype(np.float32)
    if dtype == "fp32":
        return x32, None
    bits = f32_to_bf16_bits(x32)
    return bf16_bits_to_f32(bits), bits


def _distinct_indices(seed: int, stream: int, start: int, n: int, limit: int):
    """n distinct integers in [0, limit), drawn in order from the stream."""
    chosen: list[int] = []
    pos = start
    while len(chosen) < n:
        u = uniform01(seed, stream, pos, 1)[0]
        pos += 1
        c = min(int(u * limit), limit - 1)
        if c not in chosen:
            chosen.append(c)
    return chosen, pos


def _plant_keys(seed: int, start: int, k_head: np.ndarray, n: int, scale: float,
                margin: Optional[float]):
    """n distinct keys of one head for planted rows, drawn in order from the plant stream.  With a
    margin, a candidate c is accepted only when scale * <K[c], K[c]> exceeds scale * <K[c], K[j]>
    for every other key j by more than `margin` (float64 on the stored values); duplicates and
    candidates short of the margin are skipped.  Returns (keys, next stream position, rejected
    count)."""
    n_k = k_head.shape[0]
    kh = np.asarray(k_head, dtype=np.float64) if margin is not None else None
    chosen: list[int] = []
    pos, rejected = start, 0
    for _ in range(n):
        for _attempt in range(PLANT_MAX_DRAWS):
            u = uniform01(seed, STREAM_PLANT, pos, 1)[0]
            pos += 1
            c = min(int(u * n_k), n_k - 1)
            if c in chosen:
                continue
            if margin is None:
                chosen.append(c)
                break
            sc = scale * (kh @ kh[c])
            own = sc[c]
            sc[c] = -np.inf
            if n_k == 1 or own - np.max(sc) > margin:
                chosen.append(c)
                break
            rejected += 1
        else:
            raise ValueError(f"no key with a score margin above {margin} in "
                             f"{PLANT_MAX_DRAWS} draws: this head cannot host a planted row")
    return chosen, pos, rejected


def make_inputs(cfg: AttnConfig | int) -> AttnInputs:
    if isinstance(cfg, int):
        cfg = CONFIGS[cfg]
    s = cfg.shape
    seed = cfg.the_seed
    q64 = normal(seed, STREAM_Q, s.numel_q)
    if cfg.q_sigma != 1.0:
        q64 *= cfg.q_sigma
    k64 = normal(seed, STREAM_K, s.numel_k)
    if cfg.k_sigma != 1.0:
        k64 *= cfg.k_sigma
    if cfg.v_dist == "normal":
        v64 = normal(seed, STREAM_V, s.numel_v)
    elif cfg.v_dist == "uniform":
        v64 = uniform(seed, STREAM_V, s.numel_v, -1.0, 1.0)
    else:
        raise ValueError(cfg.v_dist)
    q, qb = _store(q64, cfg.dtype)
    del q64
    k, kb = _store(k64, cfg.dtype)
    del k64
    v, vb = _store(v64, cfg.dtype)
    del v64
    q = q.reshape(s.B, s.H, s.N_q, s.d_k)
    k = k.reshape(s.B, s.H, s.N_k, s.d_k)
    v = v.reshape(s.B, s.H, s.N_k, s.d_v)
    if qb is not None:
        qb = qb.reshape(q.shape)
        kb = kb.reshape(k.shape)
        vb = vb.reshape(v.shape)
    plants = []
    redraws = 0
    if cfg.plants_per_head:
        if s.N_q < cfg.plants_per_head or s.N_k < cfg.plants_per_head:
            raise ValueError("plants need N_q, N_k >= plants_per_head")
        pos = 0
        for b in range(s.B):
            for h in range(s.H):
                rows, pos = _distinct_indices(seed, STREAM_PLANT, pos, cfg.plants_per_head, s.N_q)
                keys, pos, rej = _plant_keys(seed, pos, k[b, h], len(rows), cfg.scale,
                                             cfg.plant_margin)
                redraws += rej
                for i, kk in zip(rows, keys):
                    q[b, h, i, :] = k[b, h, kk, :]
                    if qb is not None:
                        qb[b, h, i, :] = kb[b, h, kk, :]
                    plants.append((b, h, i, kk))
    return AttnInputs(cfg, q, k, v, qb, kb, vb, tuple(plants), redraws)


def make_grad_output(cfg: AttnConfig | int, sigma: float = 1.0):
    """dL/dO for the backward pass: i.i.d. sigma * N(0,1) of O's shape [B, H, N_q, d_v], stored in
    the workload's type.  Returns (values as float32, bf16 bit patterns or None)."""
    if isinstance(cfg, int):
        cfg = CONFIGS[cfg]
    s = cfg.shape
    g64 = normal(cfg.the_seed, STREAM_DO, s.numel_o)
    if sigma != 1.0:
        g64 *= sigma
    g, gb = _store(g64, cfg.dtype)
    shape = (s.B, s.H, s.N_q, s.d_v)
    return g.reshape(shape), (gb.reshape(shape) if gb is not None else None)


def custom_config(B, H, N_q, N_k, d_k, d_v, dtype="bf16", seed=1234, q_sigma=1.0,
                  k_sigma=1.0, v_dist="normal", plants_per_head=0,
                  plant_margin=None) -> AttnConfig:
    """A workload of any shape with the same generator (used by tests)."""
    return AttnConfig(0, f"custom {dtype} B{B} H{H} Nq{N_q} Nk{N_k} dk{d_k} dv{d_v}",
                      AttnShape(B, H, N_q, N_k, d_k, d_v), dtype, q_sigma=q_sigma,
                      k_sigma=k_sigma, v_dist=v_dist, plants_per_head=plants_per_head,
                      plant_margin=plant_margin, seed=seed)
