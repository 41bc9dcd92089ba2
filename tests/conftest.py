"""pytest configuration: the `gpu` marker and shared fixtures."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


@pytest.fixture(scope="session")
def oracle():
    import oracle as _oracle
    return _oracle.get()


def load_golden(name):
    """Parse a tests/golden file: blocks of 'NAME rows cols' followed by rows."""
    import numpy as np
    path = os.path.join(ROOT, "tests", "golden", name)
    blocks = {}
    lines = [ln.split("#", 1)[0].strip() for ln in open(path)]
    lines = [ln for ln in lines if ln]
    i = 0
    while i < len(lines):
        head = lines[i].split()
        key, r, c = head[0], int(head[1]), int(head[2])
        rows = [[float(x) for x in lines[i + 1 + j].split()] for j in range(r)]
        arr = np.array(rows, dtype=np.float64)
        assert arr.shape == (r, c), (key, arr.shape)
        blocks[key] = arr
        i += 1 + r
    return blocks
