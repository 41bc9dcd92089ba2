"""The seeded input generator (shared by oracle tests and the CUDA path)."""
import numpy as np
import pytest

from paper_2606_07713_gb300 import inputs as I


def test_splitmix64_published_vector():
    # splitmix64 from state 0: first outputs of the reference generator
    # (Steele, Lea, Flood 2014; the sequence used to seed xoshiro generators).
    z = np.array([0x9E3779B97F4A7C15, (2 * 0x9E3779B97F4A7C15) % 2**64], dtype=np.uint64)
    got = I._mix64(z)
    assert int(got[0]) == 0xE220A8397B1DCDAF
    assert int(got[1]) == 0x6E789E6AA1B965F4


def test_counter_stream_is_positional():
    a = I.raw_u64(7, 2, 0, 100)
    b = I.raw_u64(7, 2, 40, 20)
    assert np.array_equal(a[40:60], b)
    assert not np.array_equal(I.raw_u64(7, 1, 0, 100), a)


def test_normal_moments():
    x = I.normal(3, 0, 1 << 20)
    assert abs(x.mean()) < 5e-3 and abs(x.std() - 1.0) < 5e-3
    assert abs(np.mean(x ** 4) - 3.0) < 0.05
    u = I.uniform(3, 2, 1 << 18, -1.0, 1.0)
    assert u.min() >= -1.0 and u.max() < 1.0 and abs(u.mean()) < 1e-2


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    x = (I.normal(11, 0, 100000) * 3).astype(np.float32)
    x[:4] = [1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -2.5, 0.0]   # ties to even, both directions
    mine = I.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(mine, ref)
    assert np.array_equal(I.bf16_bits_to_f32(mine),
                          torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_config_inputs_deterministic_and_shaped():
    cfg = I.custom_config(1, 2, 40, 70, 64, 32, dtype="bf16", seed=5, v_dist="uniform")
    a = I.make_inputs(cfg)
    b = I.make_inputs(cfg)
    assert a.q.shape == (1, 2, 40, 64) and a.k.shape == (1, 2, 70, 64) and a.v.shape == (1, 2, 70, 32)
    assert np.array_equal(a.q_bits, b.q_bits) and np.array_equal(a.v, b.v)
    assert np.array_equal(I.bf16_bits_to_f32(a.k_bits), a.k)
    assert a.v.min() >= -1.0 and a.v.max() <= 1.0


def test_plants_copy_key_rows():
    cfg = I.custom_config(1, 3, 64, 96, 128, 128, dtype="bf16", seed=9, q_sigma=8.0, k_sigma=8.0,
                          plants_per_head=4)
    x = I.make_inputs(cfg)
    assert len(x.plants) == 12
    for (b, h, i, k) in x.plants:
        assert np.array_equal(x.q_bits[b, h, i], x.k_bits[b, h, k])
    rows = {(b, h, i) for (b, h, i, _) in x.plants}
    assert len(rows) == 12


def test_five_workloads_declared():
    assert sorted(I.CONFIGS) == [1, 2, 3, 4, 5]
    s = I.CONFIGS[4].shape
    assert (s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v) == (8, 8, 1024, 4096, 128, 64)
    assert I.CONFIGS[1].dtype == "fp32" and I.CONFIGS[5].plants_per_head == 8
