"""The C-ABI library: it loads, exports every declared symbol, and its host
logic (argument and ensemble validation, the validity cut) behaves -- all
without a GPU."""
import ctypes as C

import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W


@pytest.fixture(scope="module")
def L():
    return mlt.lib()


def test_every_declared_symbol_is_exported(L):
    names = mlt.declared_symbols()
    assert {"mlt_load_ensemble", "mlt_screen", "mlt_decode_knobs", "mlt_screen_decoded",
            "mlt_screen_host", "mlt_last_error"} <= set(names)
    for name in names:
        assert hasattr(L, name), name


def test_validity_cut_matches_oracle(L):
    rng = np.random.default_rng(0)
    thrs = [0.5, 0.6, 0.1, 0.9, 0.25, 0.75, 1e-6, 0.999999, 0.5 + 2 ** -24, 0.5 - 2 ** -25]
    thrs += rng.random(200).tolist()
    for t in thrs:
        t32 = float(np.float32(t))
        if not 0.0 < t32 < 1.0:
            continue
        got = mlt.validity_cut(t32)
        want = O.tau(t32)
        assert np.float32(got).view(np.uint32) == np.float32(want).view(np.uint32), t32


@pytest.mark.parametrize("thr", [0.0, 1.0, -0.1, float("nan")])
def test_validity_cut_rejects_bad_threshold(thr):
    with pytest.raises(mlt.MltError) as e:
        mlt.validity_cut(thr)
    assert e.value.code == -1


def _stump(feature=0, thr=0.5, left=1.0, right=2.0):
    nodes = np.zeros(3, mlt.NODE_DTYPE)
    nodes[0] = (feature, thr, 1, (0, 0, 0))
    nodes[1] = (-1, left, 0, (0, 0, 0))
    nodes[2] = (-1, right, 0, (0, 0, 0))
    return nodes


def test_feature_count_bounds():
    for bad in [0, -3, 1025]:
        with pytest.raises(mlt.MltError):
            mlt.set_num_features(bad)


@pytest.mark.parametrize("case", ["unused_reachable", "feature_range", "nan_threshold", "inf_leaf",
                                  "split_at_limit", "bad_code", "overflow", "model_id", "depth",
                                  "trees"])
def test_ensemble_validation_rejects(case):
    mlt.set_num_features(4)
    nodes, n_trees, depth, model = _stump(), 1, 1, 0
    if case == "unused_reachable":
        nodes[2]["feature"] = -2
    elif case == "feature_range":
        nodes[0]["feature"] = 4
    elif case == "nan_threshold":
        nodes[0]["value"] = np.nan
    elif case == "inf_leaf":
        nodes[1]["value"] = np.inf
    elif case == "split_at_limit":
        nodes[1] = (1, 0.0, 0, (0, 0, 0))
    elif case == "bad_code":
        nodes[1]["feature"] = -7
    elif case == "overflow":
        nodes = np.concatenate([_stump(left=3e36)] * 4)
        n_trees = 4
    elif case == "model_id":
        model = 3
    elif case == "depth":
        depth = 15
        nodes = np.zeros((2 << 15) - 1, mlt.NODE_DTYPE)
    elif case == "trees":
        n_trees = 0
        nodes = nodes[:0]
    with pytest.raises((mlt.MltError, ValueError)) as e:
        mlt.load_ensemble(model, nodes, n_trees, depth)
    if isinstance(e.value, mlt.MltError):
        assert e.value.code == -1


def test_screen_rejects_bad_arguments(L):
    mlt.set_num_features(4)
    buf = C.c_void_p(16)
    # k out of range, thr out of range, negative n: rejected before any CUDA call
    assert L.mlt_screen(None, buf, 10, C.c_float(0.5), 0, buf, buf, buf) == -1
    assert L.mlt_screen(None, buf, 10, C.c_float(0.5), 16385, buf, buf, buf) == -1
    assert L.mlt_screen(None, buf, 10, C.c_float(1.5), 4, buf, buf, buf) == -1
    assert L.mlt_screen(None, buf, -1, C.c_float(0.5), 4, buf, buf, buf) == -1
    assert L.mlt_screen(None, None, 10, C.c_float(0.5), 4, buf, buf, buf) == -1
    assert L.mlt_screen(None, buf, 10, C.c_float(0.5), 0, buf, buf, buf) == -1
    assert b"k must lie" in L.mlt_last_error()


def test_decoder_validation(L):
    d = W.conv2d_decoder(seed=1)
    r = d.radices.copy()
    ov = d.option_values
    prog = d.program.copy()
    buf = C.c_void_p(16)

    def call(radices, program, first, n, F=None):
        return L.mlt_decode_knobs(None, radices.ctypes.data, ov.ctypes.data, radices.size,
                                  program.ctypes.data, program.size if F is None else F, first, n,
                                  buf, buf)

    assert call(r, prog, (1 << 24) - 4, 5) == -1  # past the end of the space
    bad = prog.copy()
    bad[10]["a"] = 8 + 10  # refers to itself
    assert call(r, bad, 0, 1) == -1
    bad = prog.copy()
    bad[3]["op"] = 12
    assert call(r, bad, 0, 1) == -1
    r2 = r.copy()
    r2[0] = 0
    assert call(r2, prog, 0, 1) == -1
    assert call(r, prog, 0, 1, F=257) == -1


@pytest.mark.parametrize("args", [(0, 48, 1, 4, 0, 0), (0, 64, 3, 4, 0, 0), (0, 256, 8, 4, 0, 0),
                                  (0, 64, 4, 3, 0, 0), (5, 64, 4, 4, 0, 0), (0, 0, 0, 0, 3, 0),
                                  (0, 0, 0, 0, 0, 4), (0, 416, 1, 4, 0, 0)])
def test_walk_tuning_rejects(args):
    with pytest.raises(mlt.MltError):
        mlt.tune_walk(*args)


def test_walk_tuning_accepts_and_releases():
    mlt.tune_walk(mlt.MLT_MODEL_P, 64, 4, 8, 8, 2)
    mlt.tune_walk(mlt.MLT_MODEL_P, 96, 2, 2, 16, 3)
    mlt.tune_walk(mlt.MLT_MODEL_V, 384, 1, 4, 4, 2)
    mlt.tune_walk(mlt.MLT_MODEL_P)
    mlt.tune_walk(mlt.MLT_MODEL_V)


@pytest.mark.parametrize("case", ["model_a", "depth_11", "leaf_past_binary16", "invalid_tree"])
def test_half_table_loader_rejects(case):
    mlt.set_num_features(4)
    nodes, n_trees, depth, model = _stump(), 1, 1, mlt.MLT_MODEL_P
    if case == "model_a":
        model = mlt.MLT_MODEL_A
    elif case == "depth_11":
        depth = 11
        nodes = np.zeros((2 << 11) - 1, mlt.NODE_DTYPE)
        nodes[0] = (-1, 0.5, 0, (0, 0, 0))
        nodes["feature"][1:] = -2
    elif case == "leaf_past_binary16":
        nodes = _stump(left=65520.0)
    elif case == "invalid_tree":
        nodes[0]["feature"] = 9
    with pytest.raises(mlt.MltError) as e:
        mlt.load_ensemble_f16(model, nodes, n_trees, depth)
    assert e.value.code == -1


@pytest.mark.parametrize("limit", [0, 999_999, 2_000_000_001])
def test_wait_selftest_rejects_limits(L, limit):
    # rejected on the host, before any CUDA call
    assert L.mlt_selftest_wait_timeout(None, limit) == -1


def test_walk_peak_rejects_bad_arguments(L):
    # rejected on the host, before any CUDA call
    mlt.set_num_features(4)
    buf = C.c_void_p(16)
    out = C.c_int64()
    assert L.mlt_walk_peak(None, 2, buf, 10, 1, buf, C.byref(out)) == -1  # model A
    assert L.mlt_walk_peak(None, 0, buf, 0, 1, buf, C.byref(out)) == -1  # n
    assert L.mlt_walk_peak(None, 0, buf, 10, 0, buf, C.byref(out)) == -1  # rounds
    assert L.mlt_walk_peak(None, 0, None, 10, 1, buf, C.byref(out)) == -1
    assert L.mlt_walk_peak(None, 0, buf, 10, 1, buf, None) == -1
    assert L.mlt_walk_peak(None, 0, buf, 10, 1, buf, C.byref(out)) == -2  # nothing loaded


@pytest.mark.parametrize("levels", [-1, 1, 5, 8, 12])
def test_head_levels_tuning_rejects(levels):
    L = mlt.lib()
    assert L.mlt_tune_head_levels(levels) == -1
    assert L.mlt_tune_head_levels(6) == 0


def test_merge_rejects_bad_arguments():
    L = mlt.lib()
    assert L.mlt_merge_topk(None, None, None, 0, 0, None) == -1  # k < 1
    assert L.mlt_merge_topk(None, None, None, -1, 5, None) == -1
    assert L.mlt_merge_topk(None, None, None, 16 * 16384 + 1, 5, None) == -1
    assert L.mlt_merge_topk(None, None, None, 10, 5, None) == -1  # NULL buffers


def test_decode_jit_tuning_and_queries():
    with pytest.raises(mlt.MltError):
        mlt.tune_decode_jit(-1)
    mlt.tune_decode_jit(0)
    mlt.tune_decode_jit(1 << 20)
    assert isinstance(mlt.decode_jit_available(), bool)
    assert mlt.decode_jit_calls() >= 0


@pytest.mark.parametrize("args", [(2, 10, 0), (5, 10, 0), (0, 0, 0), (1, -3, 1)])
def test_walk_shape_rejects(args):
    with pytest.raises(mlt.MltError):
        mlt.walk_shape(*args)
