"""Seeded synthetic screening workloads.

This module only draws inputs: candidate feature matrices, tree ensembles in
the documented heap-order node layout, and the knob space plus feature
program of the decoded conv2d workload.  It holds none of the screening
arithmetic (no tree walk, no validity decision, no decoding, no ranking);
both the CUDA library and the CPU oracle consume what it returns.

The five workloads follow the shapes of the paper's tuning tasks: candidate
schedule configurations whose features are tiling / virtual-thread knob
values plus compiler-derived hidden features (ML^2Tuner Sec. 2, Appendix A.2
"tiling and the number of virtual threads", Table 5), scored by XGBoost-style
validity and performance ensembles (Sec. 3 setup, Table 3).  Invalidity of
random configurations in the paper ranges 0.50-0.83 (Table 2), which the
survivor rates below bracket.
"""
from __future__ import annotations

import concurrent.futures
import dataclasses
import math
import os
import statistics

import numpy as np

# Documented input layouts (12-byte tree slot, 16-byte feature op).
NODE_DTYPE = np.dtype(
    [("feature", "<i4"), ("value", "<f4"), ("default_left", "u1"), ("pad", "u1", (3,))]
)
OP_DTYPE = np.dtype([("op", "<i4"), ("a", "<i4"), ("b", "<i4"), ("c", "<f4")])

LEAF = -1
UNUSED = -2

# Feature-program opcodes (operand -1 = the op's constant c).
OP_COPY, OP_ILOG2, OP_ADD, OP_SUB, OP_MUL, OP_DIV, OP_CEILDIV, OP_REM = range(8)
OP_MIN, OP_MAX, OP_GT, OP_EQ = 8, 9, 10, 11

CHUNK_ROWS = 1 << 16
THRESHOLD_SAMPLE_ROWS = 4096
LEAF_SIGMA = 0.1


@dataclasses.dataclass(frozen=True)
class ScreenConfig:
    id: int
    name: str
    n: int
    F: int
    v_trees: int
    v_depth: int
    p_trees: int
    p_depth: int
    thr: float
    k: int
    survival: float | None  # target survivor rate for the V leaf bias
    shape: str = "full"  # "full" or "unbalanced"
    split_dist: str = "uniform"  # "uniform" or "zipf"
    nan_frac: float = 0.0
    dup_frac: float = 0.0
    decoded: bool = False


CONFIGS = {
    1: ScreenConfig(1, "tiny-4096x32", 4096, 32, 50, 6, 100, 6, 0.5, 64, None),
    2: ScreenConfig(2, "gemm-65536x64", 65536, 64, 200, 8, 400, 8, 0.5, 128, 0.4),
    3: ScreenConfig(3, "sa-batch-1048576x128", 1 << 20, 128, 500, 8, 1000, 8, 0.6, 512, 0.3),
    4: ScreenConfig(4, "conv2d-exhaustive-16777216x96", 1 << 24, 96, 300, 10, 600, 10, 0.5,
                    1024, None, decoded=True),
    5: ScreenConfig(5, "skewed-nan-4194304x256", 1 << 22, 256, 1000, 12, 2000, 12, 0.5, 2048,
                    None, shape="unbalanced", split_dist="zipf", nan_frac=0.3, dup_frac=0.05),
}


@dataclasses.dataclass
class Ensemble:
    """Tree ensemble in heap order: n_trees * (2^(depth+1)-1) slots."""

    nodes: np.ndarray
    n_trees: int
    depth: int

    @property
    def slots(self) -> int:
        return (2 << self.depth) - 1


@dataclasses.dataclass
class Decoder:
    """Mixed-radix knob space plus the feature program of the decoded workload."""

    radices: np.ndarray  # int32 [n_knobs]
    option_values: np.ndarray  # float32, r_j values per knob, knob after knob
    program: np.ndarray  # OP_DTYPE [F]
    ranges: list  # per feature (lo, hi), bookkeeping for threshold draws only

    @property
    def n_knobs(self) -> int:
        return int(self.radices.size)

    @property
    def space(self) -> int:
        return int(np.prod(self.radices.astype(np.int64)))


@dataclasses.dataclass
class Workload:
    cfg: ScreenConfig
    n: int
    feats: np.ndarray | None  # [n][F] float32 (None when decoded on device)
    decoder: Decoder | None
    first_index: int
    v: Ensemble
    p: Ensemble
    thr: float
    k: int


def _rng(*key) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(x) for x in key]))


# --------------------------------------------------------------------------
# Feature matrices
# --------------------------------------------------------------------------

def _knob_cols(rng, rows, cols, n_values):
    """log2 of power-of-two knob values: integers 0 .. n_values-1."""
    return rng.integers(0, n_values, size=(rows, cols)).astype(np.float32)


def _lognormal(rng, rows, cols, sigma):
    z = rng.standard_normal(size=(rows, cols), dtype=np.float32)
    return np.exp(np.float32(sigma) * z).astype(np.float32)


def _feature_chunk(cfg: ScreenConfig, seed: int, chunk: int, rows: int) -> np.ndarray:
    rng = _rng(seed, cfg.id, 1, chunk)
    if cfg.id == 1:
        # features 0-7: log2 of {1,2,...,64}; 8-31: lognormal(0,1)
        x = np.concatenate([_knob_cols(rng, rows, 8, 7), _lognormal(rng, rows, 24, 1.0)], 1)
    elif cfg.id == 2:
        # 0-11: log2 tile/thread knobs from the divisors of 1024; 12-63:
        # lognormal(0,1.5) with 10% exact zeros
        h = _lognormal(rng, rows, 52, 1.5)
        h[rng.random(size=h.shape) < 0.1] = 0.0
        x = np.concatenate([_knob_cols(rng, rows, 12, 11), h], 1)
    elif cfg.id == 3:
        # 24 knob-derived (log2 of power-of-two divisors) + 104 lognormal(0,1)
        x = np.concatenate([_knob_cols(rng, rows, 24, 11), _lognormal(rng, rows, 104, 1.0)], 1)
    elif cfg.id == 5:
        # 16 knob-like + 240 lognormal(0,1); 30% missing (NaN); 5% duplicates
        x = np.concatenate([_knob_cols(rng, rows, 16, 11), _lognormal(rng, rows, 240, 1.0)], 1)
        x[rng.random(size=x.shape, dtype=np.float32) < cfg.nan_frac] = np.nan
        n_dup = int(round(cfg.dup_frac * rows))
        if rows > 1 and n_dup > 0:
            dst = rng.choice(rows, size=n_dup, replace=False)
            src = rng.integers(0, rows, size=n_dup)
            x[dst] = x[src]
    else:
        raise ValueError(f"workload {cfg.id} has no stored feature matrix")
    assert x.shape == (rows, cfg.F)
    return np.ascontiguousarray(x, dtype=np.float32)


def make_features(cfg: ScreenConfig, seed: int, n: int) -> np.ndarray:
    """Row-major [n][F] float32 features; rows come in fixed 65,536-row chunks,
    so a smaller n gives a prefix of the larger matrix."""
    out = np.empty((n, cfg.F), dtype=np.float32)

    def fill(c):
        a = c * CHUNK_ROWS
        b = min(n, a + CHUNK_ROWS)
        out[a:b] = _feature_chunk(cfg, seed, c, CHUNK_ROWS)[: b - a]

    chunks = range((n + CHUNK_ROWS - 1) // CHUNK_ROWS)
    if len(chunks) <= 1:
        for c in chunks:
            fill(c)
    else:
        # every chunk has its own generator (seeded by its index), so the
        # matrix does not depend on how the chunks are spread over threads
        with concurrent.futures.ThreadPoolExecutor(min(len(chunks), os.cpu_count() or 1)) as ex:
            list(ex.map(fill, chunks))
    return out


# --------------------------------------------------------------------------
# Tree ensembles
# --------------------------------------------------------------------------

def _leaf_mean(n_trees: int, thr: float, survival: float | None) -> float:
    """Per-leaf mean so that a sum of n_trees leaves N(mu, sigma) clears the
    validity threshold for about `survival` of the candidates (normal
    approximation); 0 when no rate is asked for."""
    if survival is None:
        return 0.0
    logit = math.log(thr / (1.0 - thr))
    z = statistics.NormalDist().inv_cdf(1.0 - survival)
    return (logit - LEAF_SIGMA * math.sqrt(n_trees) * z) / n_trees


def _split_features(rng, cfg: ScreenConfig, size: int) -> np.ndarray:
    if cfg.split_dist == "zipf":
        w = 1.0 / np.arange(1, cfg.F + 1, dtype=np.float64) ** 1.2
        perm = _rng(0x5EED, cfg.id, cfg.F).permutation(cfg.F)
        return perm[rng.choice(cfg.F, size=size, p=w / w.sum())].astype(np.int32)
    return rng.integers(0, cfg.F, size=size).astype(np.int32)


class _QuantileThresholds:
    """Thresholds drawn as empirical quantiles of a seeded feature sample:
    q ~ U(0,1), threshold = the floor(q*(m-1))-th order statistic of the
    non-missing values of that column."""

    def __init__(self, sample: np.ndarray):
        self.sorted = np.sort(sample, axis=0).T.copy()  # [F][m], NaN last
        self.count = np.sum(~np.isnan(sample), axis=0)

    def draw(self, rng, feats: np.ndarray) -> np.ndarray:
        q = rng.random(size=feats.size)
        m = self.count[feats]
        idx = np.floor(q * np.maximum(m - 1, 0)).astype(np.int64)
        thr = self.sorted[feats, idx]
        return np.where(m > 0, thr, 0.0).astype(np.float32)


class _RangeThresholds:
    """Thresholds for the decoded workload: drawn inside each feature's
    declared value range (log-uniform for wide positive ranges); half of them
    are rounded to an integer so that x == threshold occurs."""

    def __init__(self, ranges):
        self.lo = np.array([r[0] for r in ranges], dtype=np.float64)
        self.hi = np.array([r[1] for r in ranges], dtype=np.float64)

    def draw(self, rng, feats: np.ndarray) -> np.ndarray:
        lo, hi = self.lo[feats], self.hi[feats]
        u = rng.random(size=feats.size)
        wide = (lo > 0) & (hi > 64 * lo)
        lin = lo + u * (hi - lo)
        log = np.exp(np.log(np.maximum(lo, 1e-30)) + u * (np.log(np.maximum(hi, 1e-30)) - np.log(np.maximum(lo, 1e-30))))
        t = np.where(wide, log, lin)
        t = np.where(rng.random(size=feats.size) < 0.5, np.round(t), t)
        return t.astype(np.float32)


def make_ensemble(cfg: ScreenConfig, which: str, thresholds, seed: int, n_trees: int | None = None,
                  depth: int | None = None, split_prob: float = 0.9, shape: str | None = None) -> Ensemble:
    """Random ensemble for model 'V', 'P' or 'A' in heap order (n_trees,
    depth and shape default to the workload's V / P settings)."""
    if n_trees is None:
        n_trees = cfg.v_trees if which == "V" else cfg.p_trees
    if depth is None:
        depth = cfg.v_depth if which == "V" else cfg.p_depth
    shape = cfg.shape if shape is None else shape
    rng = _rng(seed, cfg.id, 2, {"V": 0, "P": 1, "A": 2}[which])
    slots = (2 << depth) - 1
    nodes = np.zeros((n_trees, slots), dtype=NODE_DTYPE)
    slot_depth = np.floor(np.log2(np.arange(slots) + 1)).astype(np.int64)
    if shape == "full":
        split = np.broadcast_to(slot_depth < depth, (n_trees, slots)).copy()
        leaf = ~split
    else:
        # unbalanced: the root always splits; a node at depth 1..depth-1 that
        # exists splits with probability split_prob; nodes at `depth` are leaves
        split = np.zeros((n_trees, slots), dtype=bool)
        leaf = np.zeros((n_trees, slots), dtype=bool)
        exists = np.zeros((n_trees, slots), dtype=bool)
        exists[:, 0] = True
        for d in range(depth + 1):
            a, b = (1 << d) - 1, (2 << d) - 1
            if d > 0:
                par = (np.arange(a, b) - 1) // 2
                exists[:, a:b] = split[:, par]
            if d == 0:
                s = exists[:, a:b]
            elif d < depth:
                s = exists[:, a:b] & (rng.random(size=(n_trees, b - a)) < split_prob)
            else:
                s = np.zeros((n_trees, b - a), dtype=bool)
            split[:, a:b] = s
            leaf[:, a:b] = exists[:, a:b] & ~s
    n_split = int(split.sum())
    f = _split_features(rng, cfg, n_split)
    nodes["feature"][split] = f
    nodes["value"][split] = thresholds.draw(rng, f)
    nodes["default_left"][split] = rng.integers(0, 2, size=n_split).astype(np.uint8)
    mu = _leaf_mean(n_trees, cfg.thr, cfg.survival) if which == "V" else 0.0
    n_leaf = int(leaf.sum())
    nodes["feature"][leaf] = LEAF
    nodes["value"][leaf] = (mu + LEAF_SIGMA * rng.standard_normal(size=n_leaf)).astype(np.float32)
    nodes["feature"][~(split | leaf)] = UNUSED
    return Ensemble(nodes.reshape(-1), n_trees, depth)


# --------------------------------------------------------------------------
# Decoded conv2d knob space (workload 4)
# --------------------------------------------------------------------------

class _Program:
    """Builds a feature program and tracks each feature's value range."""

    def __init__(self, knob_ranges):
        self.ops = []
        self.ranges = []
        self.n_knobs = len(knob_ranges)
        self.knob_ranges = knob_ranges

    def _rng_of(self, s, c):
        if s == -1:
            return (c, c)
        if s < self.n_knobs:
            return self.knob_ranges[s]
        return self.ranges[s - self.n_knobs]

    def slot(self, feature_index):
        return self.n_knobs + feature_index

    def add(self, op, a, b=-1, c=0.0):
        (alo, ahi), (blo, bhi) = self._rng_of(a, c), self._rng_of(b, c)
        if op in (OP_COPY,):
            r = (alo, ahi)
        elif op == OP_ILOG2:
            r = (math.floor(math.log2(max(alo, 1.0))), math.floor(math.log2(max(ahi, 1.0))))
        elif op == OP_ADD:
            r = (alo + blo, ahi + bhi)
        elif op == OP_SUB:
            r = (alo - bhi, ahi - blo)
        elif op in (OP_MUL,):
            p = [alo * blo, alo * bhi, ahi * blo, ahi * bhi]
            r = (min(p), max(p))
        elif op in (OP_DIV, OP_CEILDIV):
            assert blo > 0
            p = [alo / blo, alo / bhi, ahi / blo, ahi / bhi]
            r = (min(p), max(p))
            if op == OP_CEILDIV:
                r = (math.ceil(r[0]), math.ceil(r[1]))
        elif op == OP_REM:
            r = (0.0, min(max(ahi, 0.0), bhi))
        elif op == OP_MIN:
            r = (min(alo, blo), min(ahi, bhi))
        elif op == OP_MAX:
            r = (max(alo, blo), max(ahi, bhi))
        elif op in (OP_GT, OP_EQ):
            r = (0.0, 1.0)
        else:
            raise ValueError(op)
        self.ops.append((op, a, b, c))
        self.ranges.append((float(r[0]), float(r[1])))
        return self.slot(len(self.ops) - 1)


def conv2d_decoder(seed: int, F: int = 96) -> Decoder:
    """8 knobs x 8 power-of-two options (tile_b, tile_h, tile_w, tile_ci,
    tile_co, h_threads, w_threads, oc_nthreads) of a 3x3 convolution on a
    28x28x128 input with 128 filters, pad 1, stride 1 (ResNet18 layer shape,
    Table 2), turned into F features: knob values, their log2, tile counts and
    boundary remainders, virtual-thread counts and flags, buffer footprints
    against the extended VTA's on-chip buffers (Table 1), log-ratios, and a
    seeded tail of random combinations."""
    n_knobs, r = 8, 8
    radices = np.full(n_knobs, r, dtype=np.int32)
    option_values = np.tile(2.0 ** np.arange(r), n_knobs).astype(np.float32)
    pg = _Program([(1.0, 2.0 ** (r - 1))] * n_knobs)
    TB, TH, TW, TCI, TCO, HT, WT, OCN = range(n_knobs)
    H = W = OH = OW = 28.0
    C = KC = 128.0
    KH = KW = 3.0
    copy = [pg.add(OP_COPY, j) for j in range(n_knobs)]
    lg = [pg.add(OP_ILOG2, j) for j in range(n_knobs)]
    out_th = pg.add(OP_CEILDIV, -1, TH, OH)  # sizeOutTileH: tiles along H
    out_tw = pg.add(OP_CEILDIV, -1, TW, OW)
    bnd_h = pg.add(OP_REM, -1, TH, OH)  # boundary tile remainder
    bnd_w = pg.add(OP_REM, -1, TW, OW)
    n_filt = pg.add(OP_CEILDIV, -1, TCO, KC)  # nFilterInLoop
    n_inch = pg.add(OP_CEILDIV, -1, TCI, C)
    nvt_hw = pg.add(OP_MUL, HT, WT)
    nvt = pg.add(OP_MUL, nvt_hw, OCN)  # virtual threads
    pg.add(OP_GT, nvt, -1, 1.0)  # nVirtualThread > 1 flag
    in_h = pg.add(OP_ADD, TH, -1, KH - 1.0)  # input tile with halo
    in_w = pg.add(OP_ADD, TW, -1, KW - 1.0)
    t = pg.add(OP_MUL, TB, in_h)
    t = pg.add(OP_MUL, t, in_w)
    inp = pg.add(OP_MUL, t, TCI)  # input-buffer footprint (elements)
    t = pg.add(OP_MUL, TCO, TCI)
    wgt = pg.add(OP_MUL, t, -1, KH * KW)  # weight-buffer footprint
    t = pg.add(OP_MUL, TB, TH)
    t = pg.add(OP_MUL, t, TW)
    acc = pg.add(OP_MUL, t, TCO)  # accumulator footprint
    # extended VTA buffers (Table 1): INP 2^16 B int8, WGT 2^19 B int8,
    # ACC 2^18 B int32
    o_inp = pg.add(OP_GT, inp, -1, 2.0 ** 16)
    o_wgt = pg.add(OP_GT, wgt, -1, 2.0 ** 19)
    o_acc = pg.add(OP_GT, acc, -1, 2.0 ** 16)
    t = pg.add(OP_MAX, o_inp, o_wgt)
    pg.add(OP_MAX, t, o_acc)  # any buffer overflow
    pg.add(OP_SUB, lg[TH], lg[TW])  # log-ratios
    pg.add(OP_SUB, lg[TCI], lg[TCO])
    pg.add(OP_SUB, lg[HT], lg[WT])
    pg.add(OP_ILOG2, inp)
    pg.add(OP_ILOG2, wgt)
    pg.add(OP_ILOG2, acc)
    pg.add(OP_MIN, TH, -1, OH)  # resized output tile
    pg.add(OP_MIN, TW, -1, OW)
    t = pg.add(OP_MUL, out_th, TH)
    pg.add(OP_SUB, t, -1, OH)  # dummy rows past the output
    t = pg.add(OP_MUL, out_tw, TW)
    pg.add(OP_SUB, t, -1, OW)
    pg.add(OP_EQ, bnd_h, -1, 0.0)  # boundary tile absent
    pg.add(OP_EQ, bnd_w, -1, 0.0)
    tiles = pg.add(OP_MUL, out_th, out_tw)
    pg.add(OP_DIV, tiles, nvt_hw)  # tiles per virtual thread
    pg.add(OP_MUL, tiles, n_filt)
    pg.add(OP_DIV, inp, -1, 2.0 ** 16)  # buffer fill ratios
    pg.add(OP_DIV, acc, -1, 2.0 ** 16)
    pg.add(OP_MUL, n_inch, n_filt)
    del copy
    # seeded tail of random combinations of small-range features
    rng = _rng(seed, 4, 3)
    ops = [OP_ADD, OP_SUB, OP_MUL, OP_MIN, OP_MAX, OP_GT, OP_EQ, OP_REM]
    while len(pg.ops) < F:
        small = [s for s in range(n_knobs + len(pg.ops))
                 if (lambda r_: r_[1] - r_[0] <= 256 and r_[1] < 4096)(pg._rng_of(s, 0.0))]
        op = ops[rng.integers(len(ops))]
        a, b = (int(x) for x in rng.choice(small, size=2))
        if op == OP_REM:
            lo_b = pg._rng_of(b, 0.0)[0]
            if lo_b <= 0:
                continue
        pg.add(op, a, b)
    prog = np.zeros(F, dtype=OP_DTYPE)
    for i, (op, a, b, c) in enumerate(pg.ops[:F]):
        prog[i] = (op, a, b, c)
    return Decoder(radices, option_values, prog, pg.ranges[:F])


def make_model_a(w: "Workload", seed: int = 1, n_trees: int = 300, depth: int = 14,
                 split_prob: float = 0.75) -> Ensemble:
    """Model A for a workload: a deeper performance regressor (300 rounds,
    depth 14 in Table 3) over the same feature columns, unbalanced (a node
    below the root splits with probability split_prob), leaves N(0, 0.1)."""
    cfg = w.cfg
    if w.feats is not None:
        sample = w.feats[: min(w.n, THRESHOLD_SAMPLE_ROWS)]
        if sample.shape[0] == 0:
            sample = make_features(cfg, seed, THRESHOLD_SAMPLE_ROWS)
        th = _QuantileThresholds(sample)
    else:
        th = _RangeThresholds(w.decoder.ranges)
    return make_ensemble(cfg, "A", th, seed, n_trees=n_trees, depth=depth, split_prob=split_prob,
                         shape="unbalanced")


# --------------------------------------------------------------------------
# Whole workloads
# --------------------------------------------------------------------------

def make_workload(config_id: int, seed: int = 1, n: int | None = None) -> Workload:
    """Workload `config_id` (1-5) with `n` candidates (default: the full size)."""
    cfg = CONFIGS[int(config_id)]
    n = cfg.n if n is None else int(n)
    if cfg.decoded:
        dec = conv2d_decoder(seed, cfg.F)
        if n > dec.space:
            raise ValueError("more candidates than the knob space holds")
        th = _RangeThresholds(dec.ranges)
        feats = None
    else:
        dec = None
        feats = make_features(cfg, seed, n)
        sample = feats[: min(n, THRESHOLD_SAMPLE_ROWS)]
        if sample.shape[0] == 0:
            sample = make_features(cfg, seed, THRESHOLD_SAMPLE_ROWS)
        th = _QuantileThresholds(sample)
    v = make_ensemble(cfg, "V", th, seed)
    p = make_ensemble(cfg, "P", th, seed)
    return Workload(cfg, n, feats, dec, 0, v, p, cfg.thr, cfg.k)
