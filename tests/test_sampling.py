"""The row sample that the full-size parity tests compare when the oracle cannot afford every row
(host only)."""
import numpy as np

from gpu_helpers import SAMPLE_ROWS, sample_rows
from paper_2606_07713_gb300 import inputs as I


def test_sample_covers_every_head_first_last_and_plant():
    x = I.make_inputs(I.custom_config(2, 3, 100, 64, 64, 64, dtype="bf16", seed=2, q_sigma=8.0,
                                      k_sigma=8.0, plants_per_head=2))
    s = x.shape
    rows = sample_rows(x, n_random=60)
    assert len(rows) >= 60 and rows.max() < s.B * s.H * s.N_q
    assert set(int(r) // s.N_q for r in rows) == set(range(s.B * s.H))
    for bh in range(s.B * s.H):
        assert bh * s.N_q in rows and bh * s.N_q + s.N_q - 1 in rows
    for (b, h, i, _) in x.plants:
        assert (b * s.H + h) * s.N_q + i in rows


def test_sample_size_at_the_large_shapes():
    # the shapes of the d=128 long-sequence and stability workloads, without drawing their data
    class Fake:
        def __init__(self, shape, plants=()):
            self.shape, self.plants = shape, plants
    for shape in (I.CONFIGS[3].shape, I.CONFIGS[5].shape):
        rows = sample_rows(Fake(shape))
        per_head = np.bincount(rows // shape.N_q, minlength=shape.B * shape.H)
        assert len(rows) >= SAMPLE_ROWS
        assert per_head.min() >= SAMPLE_ROWS // (shape.B * shape.H)


def test_small_heads_are_sampled_whole():
    x = I.make_inputs(I.custom_config(1, 2, 10, 16, 64, 64, dtype="bf16", seed=4))
    assert np.array_equal(sample_rows(x), np.arange(20))
