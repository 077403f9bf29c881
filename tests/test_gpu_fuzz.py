"""GPU parity on randomly drawn screening problems.  Each case draws, from
its own seed, the feature count, the V and P tree counts, depths and shapes
(complete or unbalanced; full or compact tables), the split-feature
distribution, the feature columns (small integers, lognormal and signed
normal values, exact zeros of both signs, infinities, missing values,
duplicate rows), the batch size, the validity threshold and k, and compares
the CUDA library with the oracle: decisions, survivor counts, P scores and
top-k bit for bit, pvalid within 1e-6 relative."""
import numpy as np
import pytest

from paper_2411_10764_gb300 import workloads as W
from screening import assert_parity, assert_same_bits, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu

CASES = 40


def _features(rng, n, F, nan_frac, dup_frac):
    kinds = rng.integers(0, 3, size=F)
    cols = []
    for kind in kinds:
        if kind == 0:  # knob-like small integers (thresholds land on them)
            c = rng.integers(0, 8, size=n).astype(np.float32)
        elif kind == 1:
            c = np.exp(rng.standard_normal(n) * 1.5).astype(np.float32)
            c[rng.random(n) < 0.1] = 0.0
        else:
            c = (rng.standard_normal(n) * 3.0).astype(np.float32)
            c[rng.random(n) < 0.05] = -0.0
        cols.append(c)
    x = np.ascontiguousarray(np.stack(cols, 1), dtype=np.float32)
    clean = x.copy()  # threshold sample: finite values only
    special = rng.random(x.shape) < 0.01
    x[special] = rng.choice(np.array([np.inf, -np.inf, 0.0, -0.0], np.float32), int(special.sum()))
    if nan_frac > 0:
        x[rng.random(x.shape) < nan_frac] = np.nan
    n_dup = int(dup_frac * n)
    if n > 1 and n_dup > 0:
        x[rng.choice(n, n_dup, replace=False)] = x[rng.integers(0, n, n_dup)]
    return x, clean


def _draw_case(case):
    rng = np.random.default_rng(7000 + case)
    F = int(rng.choice([1, 3, 8, 31, 64, 97, 200, 300]))
    n = int(rng.choice([1, 7, 33, 500, 4097, 12345, 20000, 30001]))
    thr = float(rng.choice([0.05, 0.3, 0.5, 0.77, 0.97]))
    k = int(rng.choice([1, 5, 64, 300, 2049]))
    nan_frac = float(rng.choice([0.0, 0.0, 0.1, 0.5]))
    dup_frac = float(rng.choice([0.0, 0.2]))
    split_dist = str(rng.choice(["uniform", "zipf"]))
    models = []
    for which in ("V", "P"):
        shape = str(rng.choice(["full", "unbalanced"]))
        depth = int(rng.integers(1, 11)) if shape == "full" else int(rng.integers(2, 15))
        n_trees = int(rng.integers(1, 151))
        models.append((which, shape, depth, n_trees, float(rng.uniform(0.5, 0.95))))
    x, clean = _features(rng, n, F, nan_frac, dup_frac)
    cfg = W.ScreenConfig(900 + case, f"fuzz-{case}", n, F, models[0][3], models[0][2], models[1][3],
                         models[1][2], thr, k, None, split_dist=split_dist, nan_frac=nan_frac,
                         dup_frac=dup_frac)
    th = W._QuantileThresholds(clean[: min(n, 4096)])
    ens = [W.make_ensemble(cfg, which, th, 31 + case, n_trees=nt, depth=d, split_prob=sp, shape=shape)
           for which, shape, d, nt, sp in models]
    return W.Workload(cfg, n, x, None, 0, ens[0], ens[1], thr, k)


@pytest.mark.parametrize("case", range(CASES))
def test_random_problem_matches_oracle(case):
    w = _draw_case(case)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("case", range(CASES))
def test_random_problem_half_tables_match_rounded_oracle(case):
    """The same problems with binary16 tables (both models of depth <= 10):
    equal, bit for bit, to the oracle's screening of the rounded rows with the
    rounded models."""
    import torch

    import oracle as O
    from paper_2411_10764_gb300 import mlt
    from screening import THREADS

    w = _draw_case(case)
    if w.v.depth > 10 or w.p.depth > 10:
        pytest.skip("half tables hold depth <= 10")
    mlt.load_workload_models(w, half=True)
    pv, pf, tk = mlt.screen(torch.from_numpy(w.feats).cuda(), w.thr, w.k)
    mlt.sync_status()
    got = (pv.cpu().numpy(), pf.cpu().numpy(), tk.cpu().numpy(), mlt.last_survivor_count())
    x = O.round_half(w.feats)
    opv, opf, valid, _ = O.screen_rows(x, O.half_ensemble(w.v), O.half_ensemble(w.p), w.thr, threads=THREADS)
    otk, s = O.topk(opf, valid, w.k)
    assert_parity(got, (opv, opf, otk, s))


@pytest.mark.parametrize("case", range(CASES // 2))
def test_random_rerank_matches_oracle(case):
    """Model A (complete or unbalanced, depth 1 to 14, 1 to 400 trees) reranks
    a random candidate list (padding, duplicates, up to 3,000 entries) of the
    same random problems; scores bit for bit and the final order exactly."""
    import torch

    import oracle as O
    from paper_2411_10764_gb300 import mlt

    w = _draw_case(case)
    rng = np.random.default_rng(8000 + case)
    shape = str(rng.choice(["full", "unbalanced"]))
    depth = int(rng.integers(1, 11)) if shape == "full" else int(rng.integers(2, 15))
    th = W._QuantileThresholds(np.where(np.isfinite(w.feats), w.feats, np.nan)[:4096])
    a = W.make_ensemble(w.cfg, "A", th, 77 + case, n_trees=int(rng.integers(1, 401)), depth=depth,
                        split_prob=float(rng.uniform(0.5, 0.95)), shape=shape)
    m = int(rng.integers(1, 3001))
    cand = rng.integers(-1, w.n, size=m).astype(np.int64)  # -1: padding; duplicates likely
    n_final = int(rng.integers(1, m + 5))
    mlt.load_workload_models(w)
    mlt.load_ensemble(mlt.MLT_MODEL_A, a.nodes, a.n_trees, a.depth)
    sc, fin = mlt.rerank(torch.from_numpy(w.feats).cuda(), torch.from_numpy(cand).cuda(), n_final)
    mlt.sync_status()
    osc, ofin = O.rerank(w.feats, cand, a, n_final)
    assert_same_bits(sc.cpu().numpy(), osc, "A scores")
    assert np.array_equal(fin.cpu().numpy(), ofin)


def _expected_prefix(valid, n, batch, target):
    """(consumed, kept, batches) of the accumulation rule on oracle decisions."""
    kept = 0
    for b, b0 in enumerate(range(0, n, batch)):
        b1 = min(n, b0 + batch)
        kept += int(valid[b0:b1].sum())
        if kept >= target:
            return b1, kept, b + 1
    return n, kept, -(-n // batch)


@pytest.mark.parametrize("case", range(CASES // 2))
def test_random_accumulation_matches_oracle(case):
    """Batched accumulation (mlt_screen_until) over the random problems with
    random batch sizes and targets: the consumed prefix, the kept count and
    the batch count follow the accumulation rule on the oracle's decisions;
    the top-k and the prefix's scores match the oracle."""
    import torch

    import oracle as O
    from paper_2411_10764_gb300 import mlt
    from screening import THREADS, assert_pvalid

    w = _draw_case(case)
    rng = np.random.default_rng(8500 + case)
    batch = int(rng.integers(32, max(33, w.n + 100)))
    target = int(rng.integers(1, max(2, w.n)))
    mlt.load_workload_models(w)
    pv, pf, tk, stats = mlt.screen_until(torch.from_numpy(w.feats).cuda(), batch, target, w.thr, w.k)
    mlt.sync_status()
    opv, opf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    consumed, kept, batches = _expected_prefix(valid, w.n, batch, target)
    assert stats.cpu().tolist() == [consumed, kept, batches]
    want, _ = O.topk(opf[:consumed], valid[:consumed], w.k)
    assert np.array_equal(tk.cpu().numpy(), want)
    assert_same_bits(pf.cpu().numpy()[:consumed], opf[:consumed], "perf (consumed prefix)")
    assert_pvalid(pv.cpu().numpy()[:consumed], opv[:consumed])
