"""Helpers for the GPU tests: move generated inputs to the device and compare with the oracle."""
from __future__ import annotations

import numpy as np

BF16_TOL = 2e-2   # max|O - O_ref| <= BF16_TOL * max|O_ref| (bf16 inputs, fp32 accumulation)
FP32_TOL = 1e-5   # same bound for fp32 inputs


def to_device(x, dev="cuda:0"):
    """AttnInputs -> (q, k, v) torch tensors on dev in the workload's storage type."""
    import torch
    if x.cfg.dtype == "bf16":
        conv = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(dev)
        return conv(x.q_bits), conv(x.k_bits), conv(x.v_bits)
    return tuple(torch.from_numpy(np.ascontiguousarray(a)).to(dev) for a in (x.q, x.k, x.v))


def bf16_tensor_from_f32(a, dev="cuda:0"):
    """Exact bf16 tensor from float32 values that are already bf16-representable."""
    import torch
    from paper_2606_07713_gb300 import inputs as I
    bits = I.f32_to_bf16_bits(np.asarray(a, dtype=np.float32))
    assert np.array_equal(I.bf16_bits_to_f32(bits), np.asarray(a, dtype=np.float32))
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16).to(dev)


def rel_err(o_gpu: np.ndarray, o_ref: np.ndarray) -> float:
    return float(np.max(np.abs(o_gpu.astype(np.float64) - o_ref)) / np.max(np.abs(o_ref)))


def assert_close(o_gpu, o_ref, dtype: str, what: str = ""):
    tol = BF16_TOL if dtype == "bf16" else FP32_TOL
    err = rel_err(o_gpu, o_ref)
    assert np.all(np.isfinite(o_gpu)), f"{what}: non-finite output"
    assert err <= tol, f"{what}: max|O-O_ref|/max|O_ref| = {err:.3e} > {tol}"
    return err


SAMPLE_ROWS = 4096  # at least this many seeded rows where the whole output is not compared


def sample_rows(x, n_random=SAMPLE_ROWS, seed=0):
    """Flat row indices into [B*H*N_q] for sampled parity: ceil(n_random / (B*H)) distinct seeded
    rows per head (all rows of a head when it has fewer), plus the first and last row of each head
    and every planted row."""
    s = x.shape
    per_head = min(s.N_q, -(-n_random // (s.B * s.H)))
    rng = np.random.default_rng(seed)
    rows = []
    for bh in range(s.B * s.H):
        base = bh * s.N_q
        rows += [base, base + s.N_q - 1]
        rows += list(base + rng.choice(s.N_q, per_head, replace=False))
    rows += [(b * s.H + h) * s.N_q + i for (b, h, i, _) in x.plants]
    return np.unique(np.array(rows, dtype=np.int64))


def lse_bound(x, lse_ref, scale=None):
    """Per-row bound on |LSE - LSE_ref|.  A kernel forms each score in fp32 from exact products,
    so a score can be off by d_k * 2^-24 * |scale| * sum_j |q_j k_j|; the LSE, a smooth maximum of
    the scores, inherits that absolute error (4x margin), plus the relative error of the
    exp2/log2 and of the final multiply by ln 2 (4e-6 of 1 + |LSE|)."""
    scale = x.scale if scale is None else scale
    q = np.abs(x.q.astype(np.float64))
    k = np.abs(x.k.astype(np.float64))
    dk = x.q.shape[-1]
    score_err = dk * 2.0 ** -24 * abs(scale) * np.max(q @ np.swapaxes(k, -1, -2), axis=-1)
    return 4.0 * score_err + 4e-6 * (1.0 + np.abs(lse_ref))
