"""GPU parity for every launch shape of the walk kernels: results may not
depend on the shape (candidates per CTA, tree chunking, lanes per candidate,
trees in flight).  Each shape is forced through the tuning calls and
compared bit for bit with the oracle on a batch that ends on a ragged tile."""
import dataclasses

import pytest

from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import assert_parity, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu

_ORACLE = {}


def _expected(key, w):
    if key not in _ORACLE:
        _ORACLE[key] = oracle_screen(w)
    return _ORACLE[key]


@pytest.fixture(scope="module")
def deep():
    """Workload 5's shape at 3,001 candidates: 1,000 / 2,000 unbalanced trees
    of depth <= 12 on 256 features, 30 % missing values."""
    return W.make_workload(5, seed=3, n=3001)


@pytest.fixture(scope="module")
def deep_decoded():
    """The conv2d knob space with unbalanced depth-12 V and P ensembles:
    the deep walk building features from candidate indices."""
    w = W.make_workload(4, seed=2, n=3001)
    th = W._RangeThresholds(w.decoder.ranges)
    v = W.make_ensemble(w.cfg, "V", th, 5, n_trees=120, depth=12, split_prob=0.85, shape="unbalanced")
    p = W.make_ensemble(w.cfg, "P", th, 6, n_trees=200, depth=12, split_prob=0.85, shape="unbalanced")
    return dataclasses.replace(w, v=v, p=p)


@pytest.fixture(scope="module")
def full():
    return W.make_workload(2, seed=5, n=5001)


def _release():
    for m in (mlt.MLT_MODEL_V, mlt.MLT_MODEL_P):
        mlt.tune_walk(m)


def _force(**shape):
    for m in (mlt.MLT_MODEL_V, mlt.MLT_MODEL_P):
        mlt.tune_walk(m, **shape)


DEEP_SHAPES = [(c, q, g) for c in (32, 64, 128, 256) for q in (1, 2, 4, 8) for g in (4, 8) if c * q <= 256]


@pytest.mark.parametrize("cand,lanes,group", DEEP_SHAPES)
def test_compact_walk_every_shape(deep, cand, lanes, group):
    """Deep trees as compact tables (every node read through L1/L2)."""
    try:
        mlt.tune_head_levels(0)
        _force(candidates=cand, splits=lanes, group=group)
        got = gpu_screen(deep)
    finally:
        _release()
        mlt.tune_head_levels(6)
    assert_parity(got, _expected("deep", deep))


@pytest.mark.parametrize("cand,lanes,group", [(32, 8, 4), (64, 4, 8), (128, 1, 8), (32, 2, 8)])
def test_compact_walk_decoded_shapes(deep_decoded, cand, lanes, group):
    try:
        mlt.tune_head_levels(0)
        _force(candidates=cand, splits=lanes, group=group)
        got = gpu_screen(deep_decoded)
    finally:
        _release()
        mlt.tune_head_levels(6)
    assert_parity(got, _expected("deep_decoded", deep_decoded))


# split tables: (head levels, candidates per CTA, tree groups, trees in
# flight, chunk, buffers); 256 features leave room for at most 128
# candidates (F = 256) -- larger tiles fall back to the planner's choice
SPLIT_TABLE_SHAPES = ([(6, c, q, g, 8, 2) for c in (32, 64, 128) for q in (1, 2, 4) for g in (4, 8)] +
                      [(6, 64, 2, 4, ch, nb) for ch in (4, 16) for nb in (2, 3)] +
                      [(7, c, q, g, ch, 2) for c, q, g, ch in ((128, 4, 4, 16), (64, 2, 8, 16), (32, 1, 4, 4),
                                                               (128, 1, 8, 8), (128, 8, 2, 16), (32, 8, 2, 16))] +
                      [(6, 64, 8, 4, 16, 3), (6, 128, 8, 2, 8, 2), (7, 128, 4, 2, 8, 3), (6, 128, 8, 4, 32, 2),
                       (6, 64, 8, 2, 32, 2), (7, 128, 4, 2, 32, 2)])


@pytest.mark.parametrize("head,cand,groups,group,chunk,nbuf", SPLIT_TABLE_SHAPES)
def test_split_walk_every_shape(deep, head, cand, groups, group, chunk, nbuf):
    """Deep trees as split tables: the first `head` levels stream through
    shared memory, deeper nodes come from L2."""
    try:
        mlt.tune_head_levels(head)
        _force(candidates=cand, splits=groups, group=group, chunk_trees=chunk, nbuf=nbuf)
        got = gpu_screen(deep)
    finally:
        _release()
        mlt.tune_head_levels(6)
    assert_parity(got, _expected("deep", deep))


@pytest.mark.parametrize("head,cand,groups,group", [(6, 128, 4, 4), (6, 64, 1, 8), (7, 32, 2, 8), (7, 128, 2, 4),
                                                    (7, 128, 8, 2)])
def test_split_walk_decoded_shapes(deep_decoded, head, cand, groups, group):
    try:
        mlt.tune_head_levels(head)
        _force(candidates=cand, splits=groups, group=group, chunk_trees=8, nbuf=2)
        got = gpu_screen(deep_decoded)
    finally:
        _release()
        mlt.tune_head_levels(6)
    assert_parity(got, _expected("deep_decoded", deep_decoded))


FULL_SHAPES = ([(t, c, b) for t in (32, 64, 128, 256) for c in (1, 2, 4, 8, 16) for b in (2, 3)] +
               [(t, c, 2) for t in (288, 384) for c in (4, 16)])


@pytest.mark.parametrize("threads,chunk,nbuf", FULL_SHAPES)
def test_full_walk_every_shape(full, threads, chunk, nbuf):
    try:
        _force(candidates=threads, chunk_trees=chunk, nbuf=nbuf)
        got = gpu_screen(full)
    finally:
        _release()
    assert_parity(got, _expected("full", full))


# tree groups: warps of a CTA split each chunk's trees, leaves summed in order
SPLIT_SHAPES = ([(t, 2, g, c) for t in (32, 64, 96, 128) for c in (1, 4, 16) for g in (2, 4, 8)] +
                [(t, 4, g, c) for t in (32, 64) for c in (2, 8, 16) for g in (4, 8)])


@pytest.mark.parametrize("cand,splits,group,chunk", SPLIT_SHAPES)
def test_full_walk_tree_groups(full, cand, splits, group, chunk):
    try:
        _force(candidates=cand, splits=splits, group=group, chunk_trees=chunk, nbuf=2)
        got = gpu_screen(full)
    finally:
        _release()
    assert_parity(got, _expected("full", full))


@pytest.mark.parametrize("cand", [96, 160, 224, 320, 352])
def test_full_walk_candidate_counts_not_powers_of_two(full, cand):
    try:
        _force(candidates=cand)
        got = gpu_screen(full)
    finally:
        _release()
    assert_parity(got, _expected("full", full))


@pytest.fixture(scope="module")
def decoded():
    return W.make_workload(4, seed=3, n=7001)


@pytest.mark.parametrize("cand,splits,group,chunk", [(128, 2, 8, 16), (64, 4, 4, 8), (96, 2, 4, 4), (256, 1, 8, 4),
                                                     (352, 1, 4, 4), (384, 1, 2, 2)])
def test_full_walk_decoded_shapes(decoded, cand, splits, group, chunk):
    try:
        _force(candidates=cand, splits=splits, group=group, chunk_trees=chunk, nbuf=2)
        got = gpu_screen(decoded)
    finally:
        _release()
    assert_parity(got, _expected("decoded", decoded))


def test_walk_shape_reports_the_planned_and_the_forced_shape(full):
    mlt.load_workload_models(full)
    n = 1 << 20
    try:
        _force(candidates=96, splits=2, group=4, chunk_trees=8, nbuf=2)
        for p_pass in (False, True):
            sh = mlt.walk_shape(mlt.MLT_MODEL_V if not p_pass else mlt.MLT_MODEL_P, n, p_pass)
            assert (sh["candidates"], sh["splits"], sh["group"], sh["chunk_trees"], sh["nbuf"]) == (96, 2, 4, 8, 2)
            assert sh["table"] == "full"
    finally:
        _release()


def test_walk_shape_of_the_decoded_conv2d_space():
    """Depth-10 trees of 10,272 bytes beside 96 fp32 features: one CTA of 384
    candidates per SM with two 4-tree chunks, 4 trees in flight."""
    w = W.make_workload(4, seed=1, n=4096)
    mlt.load_workload_models(w)
    sh = mlt.walk_shape(mlt.MLT_MODEL_V, 1 << 24)
    assert (sh["candidates"], sh["splits"], sh["group"], sh["chunk_trees"], sh["nbuf"], sh["resident"]) == \
        (384, 1, 4, 4, 2, 1)
