import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")


def _num(v):
    if isinstance(v, str):
        return float(v)  # "nan", "inf", "-inf"
    return v


def golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def floats(seq):
    return np.array([_num(v) for v in seq], dtype=np.float32)


def slots_to_nodes(slot_lists, dtype):
    """[[feature, value, default_left], ...] (per tree) -> structured array."""
    flat = [s for tree in slot_lists for s in tree]
    out = np.zeros(len(flat), dtype=dtype)
    for i, (f, v, d) in enumerate(flat):
        out[i] = (int(f), np.float32(_num(v)), int(d), (0, 0, 0))
    return out


def same_float(a, b):
    """Bit-level equality of float32 values (NaN == NaN, -0 != +0)."""
    a = np.asarray(a, dtype=np.float32)
    b = np.asarray(b, dtype=np.float32)
    return np.array_equal(a.view(np.uint32), b.view(np.uint32))


def isclose_rel(a, b, rel):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return np.all(np.abs(a - b) <= rel * np.maximum(np.abs(b), 1e-30))
