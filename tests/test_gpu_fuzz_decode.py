"""GPU parity of the on-device knob decoder on random knob spaces and random
feature programs: every opcode; operands that are constants, knob values or
earlier features; option values and constants of both signs, zero,
subnormal and huge magnitudes (so divisions by zero, overflow to infinity and
NaN arise).  Decoded knobs and features are compared with the oracle bit for
bit (a generated NaN matches any NaN: IEEE 754 leaves its bits to the
implementation), and screening straight from candidate indices is compared
with the oracle's screening of its own decoded rows."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_parity, assert_same_bits, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu

CASES = 20
SPECIAL = np.array([0.0, -0.0, 1.0, -1.0, 2.0, 0.5, 3.0, 7.0, 1e-40, -1e-40, 1e30, -1e30, 0.1, 1024.0],
                   np.float32)


def _values(rng, size):
    v = np.where(rng.random(size) < 0.5, SPECIAL[rng.integers(0, SPECIAL.size, size)],
                 (rng.standard_normal(size) * 10.0 ** rng.integers(-3, 4, size)).astype(np.float32))
    return v.astype(np.float32)


def _decoder(case):
    rng = np.random.default_rng(9100 + case)
    n_knobs = int(rng.integers(1, 17))
    radices = rng.integers(1, 13, size=n_knobs).astype(np.int32)
    option_values = _values(rng, int(radices.sum()))
    F = int(rng.integers(1, 61))
    prog = np.zeros(F, dtype=W.OP_DTYPE)
    for f in range(F):
        prog[f]["op"] = int(rng.integers(0, 12))
        for field in ("a", "b"):
            kind = rng.integers(0, 3)
            if kind == 0 or (kind == 2 and f == 0):
                prog[f][field] = -1
            elif kind == 1:
                prog[f][field] = int(rng.integers(0, n_knobs))
            else:
                prog[f][field] = n_knobs + int(rng.integers(0, f))
        prog[f]["c"] = _values(rng, 1)[0]
    return W.Decoder(radices, option_values, prog, []), rng


@pytest.mark.parametrize("case", range(CASES))
def test_random_programs_decode_bit_exact(case):
    d, rng = _decoder(case)
    space = d.space
    n = int(min(space, rng.integers(1, 5001)))
    first = int(rng.integers(0, space - n + 1))
    knobs, feats = mlt.decode_knobs(d.radices, d.option_values, d.program, first, n)
    mlt.sync_status()
    ok, of = O.features(d.radices, d.option_values, d.program, first, n, threads=THREADS)
    assert np.array_equal(knobs.cpu().numpy(), ok)
    # every number bit for bit; a NaN the program generates matches any NaN
    assert_same_bits(feats.cpu().numpy(), of, "decoded features", nan_equal=True)
    assert np.array_equal(np.isnan(feats.cpu().numpy()), np.isnan(of))


@pytest.mark.parametrize("case", range(CASES))
def test_random_programs_screen_from_indices(case):
    d, rng = _decoder(case)
    space = d.space
    n = int(min(space, rng.integers(1, 20001)))
    first = int(rng.integers(0, space - n + 1))
    F = d.program.size
    _, sample = O.features(d.radices, d.option_values, d.program, first, min(n, 2048), threads=THREADS)
    sample = np.where(np.isfinite(sample), sample, np.nan).astype(np.float32)
    th = W._QuantileThresholds(sample)
    thr = float(rng.choice([0.2, 0.5, 0.8]))
    k = int(rng.choice([1, 16, 300]))
    cfg = W.ScreenConfig(950 + case, f"decode-fuzz-{case}", n, F, 1, 1, 1, 1, thr, k, None, decoded=True)
    shapes = [(str(rng.choice(["full", "unbalanced"])), int(rng.integers(1, 40))) for _ in range(2)]
    ens = []
    for (shape, n_trees), which in zip(shapes, ("V", "P")):
        depth = int(rng.integers(1, 9)) if shape == "full" else int(rng.integers(2, 13))
        ens.append(W.make_ensemble(cfg, which, th, 61 + case, n_trees=n_trees, depth=depth, split_prob=0.8,
                                   shape=shape))
    w = W.Workload(cfg, n, None, d, first, ens[0], ens[1], thr, k)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("case", range(6))
def test_indices_past_32_bits_decode_bit_exact(case):
    """Knob spaces of 2^35 .. 2^56 candidates (10 to 14 knobs of 12 to 16
    options): batches that straddle index 2^32, where the decoder switches
    from 32-bit to 64-bit digit division, batches at the end of the space and
    one in between."""
    d, rng = _decoder(100 + case)
    n_knobs = int(rng.integers(10, 15))
    radices = rng.integers(12, 17, size=n_knobs).astype(np.int32)
    option_values = _values(rng, int(radices.sum()))
    prog = d.program.copy()
    for f in range(prog.size):  # operands name this space's knobs
        for field in ("a", "b"):
            v = int(prog[f][field])
            if v >= d.n_knobs:
                prog[f][field] = n_knobs + (v - d.n_knobs)
            elif v >= 0:
                prog[f][field] = v % n_knobs
    d = W.Decoder(radices, option_values, prog, [])
    space = d.space
    assert space > 2 ** 34
    n = 3000
    for first in (2 ** 32 - n // 2, space - n, int(rng.integers(2 ** 33, space - n))):
        knobs, feats = mlt.decode_knobs(d.radices, d.option_values, d.program, first, n)
        mlt.sync_status()
        ok, of = O.features(d.radices, d.option_values, d.program, first, n, threads=THREADS)
        assert np.array_equal(knobs.cpu().numpy(), ok)
        assert_same_bits(feats.cpu().numpy(), of, "decoded features", nan_equal=True)


def _gpu_sa(d, parent, ps, kd, dd, lu, temperature, thr):
    import torch

    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a).astype(dt)).cuda()
    nxt, nsc, acc = mlt.sa_step(d.radices, d.option_values, d.program, t(parent, np.int64), t(ps, np.float32),
                                t(np.asarray(kd, np.uint32).view(np.int32), np.int32),
                                t(np.asarray(dd, np.uint32).view(np.int32), np.int32), t(lu, np.float32),
                                temperature, thr)
    mlt.sync_status()
    return nxt.cpu().numpy(), nsc.cpu().numpy(), acc.cpu().numpy()


@pytest.mark.parametrize("case", range(10))
def test_random_explorer_steps_match_oracle(case):
    """Three proposal steps of random chains over the random knob spaces and
    programs (random V and P ensembles on the decoded features, inactive
    chains, temperatures from hot to cold): next indices, chain scores and
    acceptances equal the oracle's."""
    d, rng = _decoder(case)
    space = d.space
    F = d.program.size
    _, sample = O.features(d.radices, d.option_values, d.program, 0, int(min(space, 2048)), threads=THREADS)
    sample = np.where(np.isfinite(sample), sample, np.nan).astype(np.float32)
    th = W._QuantileThresholds(sample)
    thr = float(rng.choice([0.3, 0.5, 0.7]))
    cfg = W.ScreenConfig(970 + case, f"sa-fuzz-{case}", 1, F, 1, 1, 1, 1, thr, 1, None, decoded=True)
    v = W.make_ensemble(cfg, "V", th, 81 + case, n_trees=int(rng.integers(1, 60)), depth=int(rng.integers(1, 9)),
                        shape="full")
    p = W.make_ensemble(cfg, "P", th, 82 + case, n_trees=int(rng.integers(1, 60)), depth=int(rng.integers(2, 13)),
                        split_prob=0.8, shape="unbalanced")
    mlt.set_num_features(F)
    mlt.load_ensemble(mlt.MLT_MODEL_V, v.nodes, v.n_trees, v.depth)
    mlt.load_ensemble(mlt.MLT_MODEL_P, p.nodes, p.n_trees, p.depth)
    m = int(rng.integers(1, 5000))
    parent = rng.integers(0, space, size=m).astype(np.int64)
    parent[rng.random(m) < 0.05] = -1  # inactive chains
    ps = np.full(m, -np.inf, np.float32)
    for step, temperature in enumerate([4.0, 1.0, 0.1]):
        kd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
        dd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
        lu = np.log(rng.random(m)).astype(np.float32)
        g = _gpu_sa(d, parent, ps, kd, dd, lu, temperature, thr)
        o = O.sa_step(d.radices, d.option_values, d.program, v, p, parent, ps, kd, dd, lu, temperature, thr)
        assert np.array_equal(g[0], o[0]), step
        assert_same_bits(g[1], o[1], f"chain scores step {step}")
        assert np.array_equal(g[2], o[2]), step
        parent, ps = o[0], o[1]
