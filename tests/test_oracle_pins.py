"""Pins of the CPU oracle against hand-worked values, closed forms, brute force
and high-precision arithmetic -- not against itself.

Paper passages: ML^2Tuner Sec. 2 (Configuration Explorer, Model V, Model P,
Model A ranking), Sec. 3 setup and Table 3 (XGBoost tree ensembles).
"""
import decimal
import itertools

import numpy as np
import pytest

import oracle as O
from conftest import floats, golden, same_float, slots_to_nodes, isclose_rel
from paper_2411_10764_gb300 import workloads as W

decimal.getcontext().prec = 60


def _f32(x):
    return float(np.float32(x))


# --------------------------------------------------------------------------
# Tree walk
# --------------------------------------------------------------------------

def test_tree_walk_hand_worked():
    g = golden("tree_walk.json")
    for tree in g["trees"]:
        nodes = slots_to_nodes([tree["slots"]], O.NODE_DTYPE)
        for row in tree["rows"]:
            got = O.tree_leaf(nodes, g["depth"], floats(row["x"]))
            assert got == row["leaf"], (tree["name"], row)


def _path_leaf(tree, depth, x):
    """Independent formulation: the reached leaf is the unique leaf slot whose
    every ancestor's condition sends x toward it."""
    slots = (2 << depth) - 1
    for leaf in range(slots):
        if tree["feature"][leaf] != -1:
            continue
        ok, j = True, leaf
        while j > 0:
            parent = (j - 1) // 2
            want_left = j == 2 * parent + 1
            f = tree["feature"][parent]
            if f < 0:
                ok = False
                break
            v, t = x[f], tree["value"][parent]
            goes_left = bool(tree["default_left"][parent]) if np.isnan(v) else bool(v < t)
            if goes_left != want_left:
                ok = False
                break
            j = parent
        if ok:
            return np.float32(tree["value"][leaf])
    raise AssertionError("no leaf reached")


@pytest.mark.parametrize("shape", ["full", "unbalanced"])
def test_margin_equals_sequential_sum_of_path_leaves(shape):
    cfg = W.ScreenConfig(99, "pin", 64, 6, 7, 4, 7, 4, 0.5, 4, None, shape=shape,
                         split_dist="uniform")
    rng = np.random.default_rng(7)
    x = rng.integers(0, 4, size=(64, 6)).astype(np.float32)  # many x == threshold
    x[rng.random(size=x.shape) < 0.2] = np.nan
    x[0, :] = np.inf
    x[1, :] = -np.inf

    class T:  # thresholds drawn from the same small integer grid
        @staticmethod
        def draw(r, f):
            return r.integers(0, 4, size=f.size).astype(np.float32)

    ens = W.make_ensemble(cfg, "V", T, seed=3)
    got = O.margins(ens, x)
    slots = ens.slots
    for i in range(x.shape[0]):
        leaves = np.array([_path_leaf(ens.nodes[t * slots:(t + 1) * slots], ens.depth, x[i])
                           for t in range(ens.n_trees)], dtype=np.float32)
        want = np.add.accumulate(np.concatenate([[np.float32(0)], leaves]), dtype=np.float32)[-1]
        assert same_float(got[i], want), i


def _stumps(left_leaves):
    """Stumps on feature 0 at 0.5 with the given left leaves (right = 0)."""
    trees = [[[0, 0.5, 1], [-1, float(l), 0], [-1, 0.0, 0]] for l in left_leaves]
    return slots_to_nodes(trees, O.NODE_DTYPE), len(trees), 1


def test_sum_is_fp32_in_tree_order():
    x = np.zeros((1, 1), np.float32)
    e = 2.0 ** -24
    # ((0 + 1) + 2^-24) + 2^-24: each add is a tie that rounds to even -> 1
    assert O.margins(_stumps([1.0, e, e]), x)[0] == 1.0
    # (2^-24 + 2^-24) + 1 = 1 + 2^-23 exactly
    assert O.margins(_stumps([e, e, 1.0]), x)[0] == 1.0 + 2.0 ** -23


def test_constant_dyadic_leaves_closed_form():
    x = np.zeros((1, 1), np.float32)
    for T, c in [(1, 0.25), (100, 0.125), (1000, -0.0625)]:
        assert O.margins(_stumps([c] * T), x)[0] == T * c


# --------------------------------------------------------------------------
# Validity decision
# --------------------------------------------------------------------------

def _sig_dec(m):
    return decimal.Decimal(1) / (decimal.Decimal(1) + (-decimal.Decimal(float(m))).exp())


@pytest.mark.parametrize("thr", [0.5, 0.6, 0.1, 0.9, 0.5 + 2 ** -24, 1e-6, 0.999999, 0.25, 0.75])
def test_tau_is_smallest_passing_float(thr):
    thr32 = np.float32(thr)
    t = np.float32(O.tau(float(thr32)))
    below = np.nextafter(t, np.float32(-np.inf))
    assert _sig_dec(t) >= decimal.Decimal(float(thr32))
    assert _sig_dec(below) < decimal.Decimal(float(thr32))


def test_tau_half_is_zero_and_invalid_thresholds():
    assert O.tau(0.5) == 0.0 and np.signbit(np.float32(O.tau(0.5))) == False  # noqa: E712
    for bad in [0.0, 1.0, -0.5, 1.5, float("nan")]:
        assert np.isnan(O.tau(bad))


def test_sigmoid_matches_high_precision():
    for m in [-20.0, -3.5, -0.75, 0.0, 0.25, 1.0, 7.0, 16.0]:
        want = float(_sig_dec(m))
        assert abs(O.sigmoid(m) - want) <= 1e-7 * want


# --------------------------------------------------------------------------
# Whole screening pass (hand-worked)
# --------------------------------------------------------------------------

def test_screen_hand_worked():
    g = golden("screen_small.json")
    v = (slots_to_nodes(g["V"], O.NODE_DTYPE), len(g["V"]), g["depth"])
    p = (slots_to_nodes(g["P"], O.NODE_DTYPE), len(g["P"]), g["depth"])
    x = np.stack([floats(r) for r in g["rows"]])
    for case in g["cases"]:
        pvalid, perf, valid, mv = O.screen_rows(x, v, p, case["thr"])
        assert same_float(mv, floats(g["margin_v"]))
        assert list(valid.astype(int)) == case["valid"]
        assert same_float(perf, floats(case["perf"]))
        assert isclose_rel(pvalid, g["pvalid"], 1e-6)
        pv2, perf2, top, s = O.screen(x, v, p, case["thr"], case["k"])
        assert s == case["survivors"]
        assert list(top) == case["topk"]
        assert same_float(perf2, perf) and same_float(pv2, pvalid)


# --------------------------------------------------------------------------
# Top-k
# --------------------------------------------------------------------------

def _brute_topk(perf, valid, k):
    order = sorted((i for i in range(len(perf)) if valid[i]), key=lambda i: (-float(perf[i]), i))
    return (order + [-1] * k)[:k], len(order)


@pytest.mark.parametrize("seed", range(6))
def test_topk_equals_first_k_of_full_sort(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(0, 300))
    perf = rng.integers(-5, 5, size=n).astype(np.float32) * np.float32(0.5)  # many ties
    perf[rng.random(size=n) < 0.1] = -0.0
    valid = rng.random(size=n) < 0.6
    for k in [1, 3, 17, 64, 400]:
        got, s = O.topk(perf, valid, k)
        want, ws = _brute_topk(perf, valid, k)
        assert s == ws and list(got) == want


def test_topk_none_valid_and_index_base():
    perf = np.array([1.0, 2.0], np.float32)
    got, s = O.topk(perf, np.zeros(2, bool), 3)
    assert s == 0 and list(got) == [-1, -1, -1]
    got, s = O.topk(perf, np.ones(2, bool), 3, index_base=100)
    assert list(got) == [101, 100, -1]


def test_screen_invariant_under_row_permutation():
    w = W.make_workload(1, seed=2, n=600)
    pv, perf, top, s = O.screen(w.feats, w.v, w.p, w.thr, 50)
    perm = np.random.default_rng(0).permutation(600)
    pv2, perf2, top2, s2 = O.screen(w.feats[perm], w.v, w.p, w.thr, 50)
    assert s == s2
    assert same_float(perf2, perf[perm]) and same_float(pv2, pv[perm])
    mapped = perm[top2[top2 >= 0]]
    kept = top[top >= 0]
    assert same_float(perf[mapped], perf[kept])  # same scores, same order
    kth = perf[kept][-1]
    assert set(kept[perf[kept] > kth]) == set(mapped[perf[mapped] > kth])


# --------------------------------------------------------------------------
# Knob decoding and feature program
# --------------------------------------------------------------------------

def test_decode_bruteforce_small_space():
    radices = [2, 3, 4]
    d = O.decode(radices, 0, 24)
    tuples = [tuple(r) for r in d]
    assert sorted(tuples) == sorted(itertools.product(range(2), range(3), range(4)))
    # knob 0 is the least significant digit (hand-worked)
    assert tuples[1] == (1, 0, 0) and tuples[2] == (0, 1, 0) and tuples[5] == (1, 2, 0)
    assert tuples[6] == (0, 0, 1) and tuples[23] == (1, 2, 3)
    for i, t in enumerate(tuples):
        assert t[0] + 2 * t[1] + 6 * t[2] == i
    assert [tuple(r) for r in O.decode(radices, 20, 4)] == tuples[20:24]
    with pytest.raises(ValueError):
        O.decode(radices, 20, 5)


def _one_op(op, a, b, c=0.0):
    prog = np.zeros(1, O.OP_DTYPE)
    prog[0] = (op, 0, 1, c)
    _, f = O.features([1, 1], np.array([a, b], np.float32), prog, 0, 1)
    return f[0, 0]


def test_feature_ops_hand_worked():
    g = golden("feature_ops.json")
    for name, a, b, want, why in g["cases"]:
        got = _one_op(g["ops"][name], *floats([a, b]))
        assert same_float(got, floats([want])[0]), (name, a, b, why)


def test_feature_program_constants_and_earlier_features():
    prog = np.zeros(3, O.OP_DTYPE)
    prog[0] = (W.OP_CEILDIV, -1, 0, 28.0)  # ceil(28 / knob0)
    prog[1] = (W.OP_ADD, 1 + 0, 1 + 0, 0.0)  # feature0 + feature0
    prog[2] = (W.OP_SUB, 1 + 1, -1, 1.0)  # feature1 - 1
    _, f = O.features([3], np.array([8.0, 4.0, 128.0], np.float32), prog, 0, 3)
    assert f.tolist() == [[4.0, 8.0, 7.0], [7.0, 14.0, 13.0], [1.0, 2.0, 1.0]]
    bad = prog.copy()
    bad[1] = (W.OP_ADD, 3, 0, 0.0)  # refers to a feature not yet computed
    with pytest.raises(ValueError):
        O.features([3], np.array([8.0, 4.0, 128.0], np.float32), bad, 0, 1)


def test_conv2d_features_hand_worked():
    g = golden("conv2d_features.json")
    dec = W.conv2d_decoder(seed=1)
    assert dec.radices.tolist() == [g["radix"]] * 8
    for case in g["cases"]:
        knobs, f = O.features(dec.radices, dec.option_values, dec.program, case["index"], 1)
        assert knobs[0].tolist() == case["digits"]
        assert same_float(f[0, :60], np.array(case["features_0_59"], np.float32)), case["index"]


# --------------------------------------------------------------------------
# Model A rerank
# --------------------------------------------------------------------------

def test_rerank_hand_worked():
    g = golden("screen_small.json")
    a = (slots_to_nodes(g["A"], O.NODE_DTYPE), len(g["A"]), g["A_depth"])
    x = np.stack([floats(r) for r in g["rows"]])
    for case in g["rerank_cases"]:
        score, final = O.rerank(x, g["rerank_cand"], a, case["n_final"])
        assert same_float(score, floats(g["rerank_score"]))
        assert final.tolist() == case["final"]


@pytest.mark.parametrize("seed", range(4))
def test_rerank_equals_sorted_margins(seed):
    rng = np.random.default_rng(seed)
    w = W.make_workload(1, seed=seed + 1, n=500)
    cand = rng.choice(500, size=40, replace=False).astype(np.int64)
    cand[rng.random(40) < 0.2] = -1
    score, final = O.rerank(w.feats, cand, w.p, 25)
    m = O.margins(w.p, w.feats)
    valid = [int(c) for c in cand if c >= 0]
    want = sorted(valid, key=lambda c: (-float(m[c]), c))[:25]
    assert final.tolist() == want + [-1] * (25 - len(want))
    for i, c in enumerate(cand):
        assert same_float(score[i], m[c] if c >= 0 else np.float32(-np.inf))


# --------------------------------------------------------------------------
# Explorer proposal step
# --------------------------------------------------------------------------

def _sa_fixture():
    g = golden("sa_step.json")
    prog = np.zeros(len(g["program"]), O.OP_DTYPE)
    for i, (op, a, b, c) in enumerate(g["program"]):
        prog[i] = (op, a, b, c)
    v = (slots_to_nodes(g["V"], O.NODE_DTYPE), len(g["V"]), g["depth"])
    p = (slots_to_nodes(g["P"], O.NODE_DTYPE), len(g["P"]), g["depth"])
    return g, prog, v, p


def test_sa_step_hand_worked():
    g, prog, v, p = _sa_fixture()
    for case in g["cases"]:
        nxt, nsc, acc = O.sa_step(g["radices"], g["options"], prog, v, p, g["parent"], floats(g["parent_score"]),
                                  g["knob_draw"], g["digit_draw"], floats(g["log_u"]), case["temperature"], g["thr"])
        assert nxt.tolist() == case["next"]
        assert same_float(nsc, floats(case["score"]))
        assert acc.tolist() == case["accepted"]


def test_sa_step_proposals_change_one_knob():
    d = W.conv2d_decoder(seed=1)
    w = W.make_workload(4, seed=1, n=2000)
    rng = np.random.default_rng(3)
    m = 300
    parent = rng.integers(0, d.space, size=m)
    ps = np.full(m, -np.inf, np.float32)  # every valid proposal is accepted
    kd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
    dd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
    lu = np.log(rng.random(m)).astype(np.float32)
    nxt, nsc, acc = O.sa_step(d.radices, d.option_values, d.program, w.v, w.p, parent, ps, kd, dd, lu, 1.0, w.thr)
    pk = O.decode(d.radices, 0, 1)  # warm the library
    for i in range(m):
        a = O.decode(d.radices, int(parent[i]), 1)[0]
        j = int(kd[i]) % 8
        q = a.copy()
        q[j] = int(dd[i]) % 8
        qi = int(sum(int(q[t]) * 8 ** t for t in range(8)))
        if acc[i]:
            assert nxt[i] == qi
            _, f = O.features(d.radices, d.option_values, d.program, qi, 1)
            _, pf, valid, _ = O.screen_rows(f, w.v, w.p, w.thr)
            assert valid[0] and same_float(nsc[i], pf[0])
        else:
            assert nxt[i] == parent[i] and np.isneginf(nsc[i])
    del pk


# ---------------------------------------------------------------------------
# Half tables: the binary16 rounding the variant applies (IEEE 754 binary16:
# 1 sign, 5 exponent, 10 fraction bits; round to nearest, ties to even).
# Expected values worked by hand from that definition.
# ---------------------------------------------------------------------------
HALF_CASES = [
    (1.0, 1.0),
    (0.1, 0.0999755859375),              # 0x2E66: 1638/16384
    (1.0 + 2.0 ** -11, 1.0),             # tie between 1 and 1 + 2^-10: even fraction wins
    (1.0 + 3 * 2.0 ** -11, 1.0 + 2.0 ** -9),  # tie between fractions 1 and 2: 2 is even
    (1.0 + 2.0 ** -11 + 2.0 ** -20, 1.0 + 2.0 ** -10),  # just above the tie
    (65504.0, 65504.0),                  # largest finite
    (65519.0, 65504.0),
    (65520.0, np.inf),                   # the tie with 2^16 rounds to infinity
    (-70000.0, -np.inf),
    (2.0 ** -24, 2.0 ** -24),            # smallest subnormal
    (2.0 ** -25, 0.0),                   # tie with 0: even (0) wins
    (3 * 2.0 ** -26, 2.0 ** -24),
    (-0.0, -0.0),
    (1025.0, 1025.0),                    # spacing is 1 in [1024, 2048)
    (2049.0, 2048.0),                    # spacing 2 in [2048, 4096): tie, 2048 is even
    (2051.0, 2052.0),                    # tie between 2050 and 2052: 2052 is even
]


@pytest.mark.parametrize("x,expect", HALF_CASES)
def test_round_half_hand_worked(x, expect):
    got = O.round_half(np.float32(x))
    assert got.dtype == np.float32
    assert float(got) == expect and np.signbit(got) == np.signbit(np.float64(expect))


def test_round_half_keeps_nan_and_infinities():
    got = O.round_half(np.array([np.nan, np.inf, -np.inf], np.float32))
    assert np.isnan(got[0]) and got[1] == np.inf and got[2] == -np.inf


def test_round_half_is_monotone_and_idempotent():
    rng = np.random.default_rng(7)
    x = np.sort(rng.standard_normal(100000).astype(np.float32) * rng.choice([1e-3, 1.0, 1e3], 100000))
    h = O.round_half(x)
    assert np.all(np.diff(h.astype(np.float64)) >= 0)
    assert np.array_equal(O.round_half(h), h)


def test_half_ensemble_rounds_values_only():
    w = W.make_workload(2, seed=1, n=1000)
    nodes, n_trees, depth = O.half_ensemble(w.v)
    assert (n_trees, depth) == (w.v.n_trees, w.v.depth)
    assert np.array_equal(nodes["feature"], w.v.nodes["feature"])
    assert np.array_equal(nodes["default_left"], w.v.nodes["default_left"])
    used = nodes["feature"] != W.UNUSED
    assert np.array_equal(nodes["value"][used], O.round_half(w.v.nodes["value"][used]))
    assert np.array_equal(nodes["value"][~used], w.v.nodes["value"][~used])
