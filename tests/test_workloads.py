"""Seeded workload generators: determinism, shapes and structure."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import workloads as W


def _check_heap(ens: W.Ensemble, F: int):
    t = ens.nodes.reshape(ens.n_trees, ens.slots)
    feat = t["feature"]
    depth_of = np.floor(np.log2(np.arange(ens.slots) + 1)).astype(int)
    assert np.all(feat[:, 0] != W.UNUSED)
    for j in range(ens.slots):
        split = feat[:, j] >= 0
        if depth_of[j] == ens.depth:
            assert not split.any()
            continue
        l, r = 2 * j + 1, 2 * j + 2
        assert np.all(feat[split, l] != W.UNUSED) and np.all(feat[split, r] != W.UNUSED)
        not_split = ~split
        assert np.all(feat[not_split, l] == W.UNUSED) and np.all(feat[not_split, r] == W.UNUSED)
    assert feat.max() < F
    vals = t["value"][feat != W.UNUSED]
    assert np.all(np.isfinite(vals))


@pytest.mark.parametrize("cid", [1, 2, 3, 5])
def test_small_workloads_are_deterministic_and_well_formed(cid):
    a = W.make_workload(cid, seed=1, n=3000)
    b = W.make_workload(cid, seed=1, n=3000)
    c = W.make_workload(cid, seed=2, n=3000)
    assert a.feats.shape == (3000, a.cfg.F) and a.feats.dtype == np.float32
    assert np.array_equal(a.feats, b.feats, equal_nan=True)
    assert not np.array_equal(a.feats, c.feats, equal_nan=True)
    assert np.array_equal(a.v.nodes, b.v.nodes) and np.array_equal(a.p.nodes, b.p.nodes)
    _check_heap(a.v, a.cfg.F)
    _check_heap(a.p, a.cfg.F)
    assert a.v.n_trees == a.cfg.v_trees and a.p.n_trees == a.cfg.p_trees


def test_feature_rows_are_a_prefix_across_sizes():
    small = W.make_features(W.CONFIGS[2], 1, 1000)
    large = W.make_features(W.CONFIGS[2], 1, 70000)
    assert np.array_equal(small, large[:1000])


def test_workload5_missing_values_duplicates_and_tree_size():
    w = W.make_workload(5, seed=1, n=65536)
    assert 0.28 < np.isnan(w.feats).mean() < 0.32
    _, counts = np.unique(w.feats.view(np.uint32).reshape(65536, -1), axis=0, return_counts=True)
    dup_rows = counts[counts > 1].sum()
    assert 0.03 * 65536 < dup_rows < 0.12 * 65536
    per_tree = (w.v.nodes["feature"] != W.UNUSED).sum() / w.v.n_trees
    assert 2600 < per_tree < 3200  # about 2,890 nodes per tree


def test_workload2_knob_features_and_zeros():
    x = W.make_features(W.CONFIGS[2], 1, 20000)
    knobs = x[:, :12]
    assert set(np.unique(knobs).tolist()) == set(float(i) for i in range(11))
    assert 0.08 < (x[:, 12:] == 0).mean() < 0.12


@pytest.mark.parametrize("cid,lo,hi", [(1, 0.2, 0.8), (2, 0.3, 0.5), (3, 0.2, 0.4)])
def test_survivor_rates_near_targets(cid, lo, hi):
    w = W.make_workload(cid, seed=1, n=4096)
    _, _, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=4)
    assert lo < valid.mean() < hi


def test_conv2d_decoder_program_is_well_formed():
    d = W.conv2d_decoder(seed=1)
    assert d.program.size == 96 and d.space == 1 << 24
    for i, (op, a, b, c) in enumerate(d.program.tolist()):
        assert 0 <= op <= 11
        assert -1 <= a < 8 + i and -1 <= b < 8 + i
