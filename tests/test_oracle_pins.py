"""The fp64 oracle against what the paper and mathematics fix (CPU only)."""
import numpy as np
import pytest

import oracle_pins


@pytest.mark.parametrize("pin", oracle_pins.ALL_PINS, ids=lambda f: f.__name__)
def test_oracle_pin(oracle, pin):
    pin(oracle)


def test_oracle_rejects_bad_arguments(oracle):
    q = np.zeros((1, 1, 2, 4), np.float32)
    k = np.zeros((1, 1, 0, 4), np.float32)
    v = np.zeros((1, 1, 0, 4), np.float32)
    with pytest.raises(RuntimeError):
        oracle.attn(q, k, v, 1.0)
    with pytest.raises(RuntimeError):
        oracle.rows(q, np.zeros((1, 1, 3, 4), np.float32), np.zeros((1, 1, 3, 4), np.float32),
                    1.0, [5])


def test_oracle_threads_reported(oracle):
    assert oracle.max_threads() >= 1
