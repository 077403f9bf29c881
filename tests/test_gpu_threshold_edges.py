"""GPU parity of the node test `x < threshold` at its edges: feature values on
thresholds, one or two ulps away, and 4095 / 4096 / 4097 / 8192 / 100000
ulps away (counted in the order of the floats, so across +-0 too), on
thresholds that are small integers and powers of two (the knob features'
values) and on unaligned ones, on +-0, subnormals, +-FLT_MAX, infinities and
NaN with both default sides -- all against the oracle, bit for bit."""
import dataclasses

import numpy as np
import pytest

from paper_2411_10764_gb300 import workloads as W
from screening import assert_parity, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu

F32 = np.float32
MAXF = np.finfo(F32).max
TINY = np.float32(1e-45)  # smallest subnormal


def to_key(x):
    """Position of float32 values in the order of the floats (-0 on +0)."""
    u = np.asarray(x, F32).view(np.uint32).astype(np.uint64)
    k = np.where(u & 0x80000000, ~u & 0xFFFFFFFF, u | 0x80000000)
    return np.where(np.asarray(x, F32) == 0, 0x80000000, k).astype(np.uint64)


def from_key(k):
    k = np.asarray(k, np.uint64)
    u = np.where(k & 0x80000000, k & 0x7FFFFFFF, ~k & 0xFFFFFFFF).astype(np.uint32)
    return u.view(F32)


def shifted(thr, d):
    """thr moved by d positions in the order of the floats, kept finite."""
    k = to_key(thr).astype(np.int64) + d
    lo, hi = int(to_key(-MAXF)), int(to_key(MAXF))
    return from_key(np.clip(k, lo, hi).astype(np.uint64))


SHIFTS = np.array([0, 1, -1, 2, -2, 4095, -4095, 4096, -4096, 4097, -4097, 8192, -8192, 100000, -100000])
SPECIAL_X = np.array([np.nan, np.inf, -np.inf, 0.0, -0.0, TINY, -TINY, MAXF, -MAXF], F32)
# thresholds with many trailing zero mantissa bits, unaligned ones, +-0, extremes
SPECIAL_THR = np.array([0.0, -0.0, 1.0, 2.0, 3.0, 0.5, -1.0, -7.0, 1024.0, 1.0000001, 0.3, -0.3,
                        3.1415927, TINY, -TINY, MAXF, -MAXF, 1e-38, -1e-38, 65536.5], F32)


class _SpecialThresholds:
    def draw(self, rng, feats):
        return SPECIAL_THR[rng.integers(0, SPECIAL_THR.size, size=feats.size)]


def _near_thresholds(w, x, rng, n_edits, shifts=SHIFTS):
    """Put n_edits feature values at thresholds of the V and P ensembles moved
    by the given shifts, and some special values."""
    nodes = np.concatenate([w.v.nodes, w.p.nodes])
    split = nodes["feature"] >= 0
    thr, feat = nodes["value"][split], nodes["feature"][split]
    rows = rng.integers(0, x.shape[0], n_edits)
    pick = rng.integers(0, thr.size, n_edits)
    x[rows, feat[pick]] = shifted(thr[pick], shifts[rng.integers(0, shifts.size, n_edits)])
    r2 = rng.integers(0, x.shape[0], n_edits // 10)
    c2 = rng.integers(0, x.shape[1], n_edits // 10)
    x[r2, c2] = SPECIAL_X[rng.integers(0, SPECIAL_X.size, r2.size)]
    return x


def test_shift_helpers_round_trip():
    v = np.array([0.0, 1.0, -1.0, 3.5, -MAXF, MAXF, TINY, -TINY, 1e-38], F32)
    assert np.array_equal(from_key(to_key(v)).view(np.uint32), v.view(np.uint32))
    assert shifted(np.array([1.0], F32), 1)[0] == np.nextafter(F32(1.0), F32(2.0))
    assert shifted(np.array([TINY], F32), -1)[0] == 0.0


@pytest.mark.parametrize("cid,n,seed", [(2, 6000, 1), (3, 5000, 2), (1, 4096, 3)])
def test_features_at_and_near_thresholds(cid, n, seed):
    w = W.make_workload(cid, seed=seed, n=n)
    x = _near_thresholds(w, w.feats.copy(), np.random.default_rng(seed), n * 4)
    assert_parity(gpu_screen(w, feats=x), oracle_screen(w, feats=x))


@pytest.mark.parametrize("depth,shape", [(3, "full"), (8, "full"), (10, "unbalanced")])
def test_special_thresholds(depth, shape):
    """Thresholds drawn only from round, unaligned and extreme values;
    features on and around them, and NaN with both default sides."""
    w = W.make_workload(2, seed=9, n=7001)
    th = _SpecialThresholds()
    v = W.make_ensemble(w.cfg, "V", th, 21, n_trees=60, depth=depth, split_prob=0.8, shape=shape)
    p = W.make_ensemble(w.cfg, "P", th, 22, n_trees=120, depth=depth, split_prob=0.8, shape=shape)
    w = dataclasses.replace(w, v=v, p=p, thr=0.3)
    rng = np.random.default_rng(depth)
    x = SPECIAL_THR[rng.integers(0, SPECIAL_THR.size, w.feats.shape)]
    x = shifted(x.ravel(), SHIFTS[rng.integers(0, SHIFTS.size, x.size)]).reshape(w.feats.shape).copy()
    mask = rng.random(x.shape) < 0.05
    x[mask] = SPECIAL_X[rng.integers(0, SPECIAL_X.size, int(mask.sum()))]
    x = np.ascontiguousarray(x, F32)
    assert_parity(gpu_screen(w, feats=x), oracle_screen(w, feats=x))


def test_decoded_features_near_thresholds():
    """The decoding walk computes the features on the device: move every
    threshold onto a small integer (what knob-derived features take) or the
    float next to one."""
    w = W.make_workload(4, seed=5, n=20000)
    rng = np.random.default_rng(5)

    def snap(ens):
        nodes = ens.nodes.copy()
        split = nodes["feature"] >= 0
        thr = nodes["value"][split]
        k = rng.integers(0, 3, thr.size)
        nodes["value"][split] = np.where(k == 0, np.round(thr), np.where(k == 1, shifted(np.round(thr), 1),
                                                                            shifted(np.round(thr), -1)))
        return dataclasses.replace(ens, nodes=nodes)

    w = dataclasses.replace(w, v=snap(w.v), p=snap(w.p))
    assert_parity(gpu_screen(w), oracle_screen(w))
