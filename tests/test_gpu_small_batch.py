"""The single-launch path for small batches (one kernel: V walk, validity, P
walk, rank keys and the top-k selection by its last CTA) against the oracle
and against the four-kernel path, bit for bit: shapes that take it (full V
and P tables of one depth, up to 8,192 candidates), every branch of its
selection (up to 512 survivors ranked directly, the k-th key's bucket
collected and ranked, a crowded bucket sorted whole), and shapes that do
not take it."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_parity, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu


def _both_paths(w, k=None, feats=None):
    """(single-launch result, four-kernel result)."""
    try:
        mlt.tune_fused_small(8192)
        fused = gpu_screen(w, k=k, feats=feats)
        mlt.tune_fused_small(0)
        multi = gpu_screen(w, k=k, feats=feats)
    finally:
        mlt.tune_fused_small(8192)
    return fused, multi


def _same(a, b):
    for x, y in zip(a[:3], b[:3]):
        x, y = np.asarray(x), np.asarray(y)
        if x.dtype == np.float32:
            assert np.array_equal(x.view(np.uint32), y.view(np.uint32))
        else:
            assert np.array_equal(x, y)
    assert a[3] == b[3]


@pytest.mark.parametrize("cid,n,k", [(1, 4096, 64), (1, 1, 8), (1, 33, 5), (2, 5000, 128), (2, 8192, 700),
                                     (2, 8192, 16384), (1, 300, 64), (1, 4097, 512)])
def test_single_launch_matches_oracle_and_four_kernel_path(cid, n, k):
    w = W.make_workload(cid, seed=11, n=n)
    fused, multi = _both_paths(w, k=k)
    assert_parity(fused, oracle_screen(w, k=k))
    _same(fused, multi)


@pytest.mark.parametrize("k", [1, 100, 512, 513, 4000, 8000, 8192])
def test_single_launch_crowded_bucket(k):
    """8,000 copies of one surviving candidate: every key shares its score,
    so the k-th key's bucket holds them all and the last CTA sorts every
    key; ties go to the smaller index."""
    w = W.make_workload(2, seed=1, n=2000)
    _, _, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    row = w.feats[int(np.nonzero(valid)[0][0])]
    x = np.ascontiguousarray(np.tile(row, (8000, 1)))
    fused, multi = _both_paths(w, k=k, feats=x)
    opv, opf, otk, os_ = oracle_screen(w, feats=x, k=k)
    assert os_ == 8000
    assert_parity(fused, (opv, opf, otk, os_))
    _same(fused, multi)


def test_single_launch_with_missing_values_and_unaligned_width():
    cfg = W.ScreenConfig(97, "f30", 3000, 30, 40, 6, 50, 6, 0.5, 64, None)
    x = W.make_features(W.CONFIGS[1], 3, 3000)
    x = np.ascontiguousarray(np.tile(x, (1, 2))[:, :30])
    rng = np.random.default_rng(3)
    x[rng.random(size=x.shape) < 0.2] = np.nan
    th = W._QuantileThresholds(x[:2048])
    w = W.Workload(cfg, 3000, x, None, 0, W.make_ensemble(cfg, "V", th, 5), W.make_ensemble(cfg, "P", th, 6), 0.5, 64)
    fused, multi = _both_paths(w)
    assert_parity(fused, oracle_screen(w))
    _same(fused, multi)


def test_models_of_different_depths_take_the_four_kernel_path():
    cfg = W.ScreenConfig(96, "mixed", 2000, 32, 30, 6, 40, 8, 0.5, 50, None)
    x = W.make_features(W.CONFIGS[1], 4, 2000)
    th = W._QuantileThresholds(x[:2048])
    w = W.Workload(cfg, 2000, x, None, 0, W.make_ensemble(cfg, "V", th, 7), W.make_ensemble(cfg, "P", th, 8), 0.5, 50)
    launches = mlt.kernel_launches()
    g = gpu_screen(w)
    assert mlt.kernel_launches() - launches == 4
    assert_parity(g, oracle_screen(w))


def test_single_launch_is_one_kernel():
    w = W.make_workload(1, seed=2, n=4096)
    mlt.load_workload_models(w)
    import torch

    x = torch.from_numpy(w.feats).cuda()
    launches = mlt.kernel_launches()
    mlt.screen(x, w.thr, w.k)
    mlt.sync_status()
    assert mlt.kernel_launches() - launches == 1
