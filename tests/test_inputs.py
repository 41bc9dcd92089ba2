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


def test_stress_workload_declares_the_margin():
    assert I.CONFIGS[5].plant_margin == I.PLANT_MARGIN == 30.0
    assert all(I.CONFIGS[c].plant_margin is None for c in (1, 2, 3, 4))


def test_five_workloads_declared():
    assert sorted(I.CONFIGS) == [1, 2, 3, 4, 5]
    s = I.CONFIGS[4].shape
    assert (s.B, s.H, s.N_q, s.N_k, s.d_k, s.d_v) == (8, 8, 1024, 4096, 128, 64)
    assert I.CONFIGS[1].dtype == "fp32" and I.CONFIGS[5].plants_per_head == 8


def _margins(oracle, x):
    """Score margin of every planted row over its next-best key, from the oracle's scores."""
    out = []
    for (b, h, i, kk) in x.plants:
        sc = oracle.scores(x.q[b, h, i:i + 1], x.k[b, h], x.scale)[0]
        own = sc[kk]
        sc[kk] = -np.inf
        out.append(own - np.max(sc))
    return np.array(out)


def test_plant_keys_redrawn_until_margin(oracle):
    # Q, K ~ 2.5 N(0,1), d = 64, 1024 keys: a planted score is about 50 +- 9 and the next best
    # about 20, so roughly half of the first candidates fall short of the margin and are redrawn.
    cfg = I.custom_config(1, 3, 64, 1024, 64, 64, dtype="bf16", seed=9, q_sigma=2.5, k_sigma=2.5,
                          plants_per_head=4, plant_margin=I.PLANT_MARGIN)
    x = I.make_inputs(cfg)
    assert x.plant_redraws > 0
    assert np.all(_margins(oracle, x) > I.PLANT_MARGIN)
    for h in range(3):
        keys = [kk for (_, hh, _, kk) in x.plants if hh == h]
        rows = [i for (_, hh, i, _) in x.plants if hh == h]
        assert len(set(keys)) == 4 and len(set(rows)) == 4
    # the redraws come from the seeded stream, so the plants are reproducible
    y = I.make_inputs(cfg)
    assert y.plants == x.plants
    # without a margin the first distinct candidates are kept, some of them short of it
    z = I.make_inputs(I.custom_config(1, 3, 64, 1024, 64, 64, dtype="bf16", seed=9, q_sigma=2.5,
                                      k_sigma=2.5, plants_per_head=4))
    assert z.plant_redraws == 0 and np.min(_margins(oracle, z)) < I.PLANT_MARGIN


def test_plant_margin_holds_for_stress_shape(oracle):
    # the stability workload's distributions (sigma 8, d = 128) at a smaller key count
    cfg = I.custom_config(1, 2, 256, 4096, 128, 128, dtype="bf16", seed=5, q_sigma=8.0,
                          k_sigma=8.0, plants_per_head=8, plant_margin=I.PLANT_MARGIN)
    x = I.make_inputs(cfg)
    assert len(x.plants) == 16 and np.all(_margins(oracle, x) > I.PLANT_MARGIN)


def test_plant_without_any_margin_is_refused():
    # d = 8, unit scale: a planted score is about 2.8, far below the margin for every key
    cfg = I.custom_config(1, 1, 16, 64, 8, 8, dtype="fp32", seed=3, plants_per_head=1,
                          plant_margin=I.PLANT_MARGIN)
    with pytest.raises(ValueError, match="margin"):
        I.make_inputs(cfg)
