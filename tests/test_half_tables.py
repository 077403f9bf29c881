"""The half-table variant's tolerance, checked on the oracle alone: how far
the binary16-rounded model (rounded thresholds, leaves and features) moves
the screening results away from the fp32 model on the synthetic workloads.
The CUDA half tables are pinned to the rounded model bit for bit by the GPU
tests; these bounds are what a user of the variant trades for its speed."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import workloads as W

THREADS = 8


def _both(cid, n):
    w = W.make_workload(cid, seed=1, n=n)
    exact = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    rounded = O.screen_rows(O.round_half(w.feats), O.half_ensemble(w.v), O.half_ensemble(w.p), w.thr,
                            threads=THREADS)
    return w, exact, rounded


@pytest.mark.parametrize("cid,n", [(1, 4096), (2, 20000), (3, 6000)])
def test_rounded_model_tolerance(cid, n):
    w, (_, pf, valid, _), (_, pf_h, valid_h, _) = _both(cid, n)
    # validity decisions: at most 1 % flip
    assert (valid != valid_h).mean() <= 0.01
    # scores of candidates valid under both: median shift below 1e-2, all
    # below 1 (the scores span several units)
    both = valid & valid_h
    d = np.abs(pf_h[both].astype(np.float64) - pf[both])
    assert np.median(d) <= 1e-2 and d.max() < 1.0
    # the kept set: at least 95 % of the exact top-k is kept, and at least
    # 98 % of the rounded top-k lies in the exact top-2k
    tk, _ = O.topk(pf, valid, w.k)
    tk_h, _ = O.topk(pf_h, valid_h, w.k)
    assert len(set(tk.tolist()) & set(tk_h.tolist())) >= 0.95 * w.k
    tk2, _ = O.topk(pf, valid, 2 * w.k)
    assert len(set(tk_h.tolist()) & set(tk2.tolist())) >= 0.98 * w.k


def test_rounded_model_is_exact_on_representable_inputs():
    """Knob-like features (small integers) and thresholds that binary16
    holds exactly: the rounded model must equal the fp32 model."""
    w = W.make_workload(1, seed=2, n=3000)
    feats = np.round(w.feats * 4) / 4                      # quarter steps: exact in binary16
    feats = np.clip(feats, -1000, 1000).astype(np.float32)
    v = O.half_ensemble(w.v)                               # the model is now representable
    p = O.half_ensemble(w.p)
    a = O.screen_rows(feats, v, p, w.thr, threads=THREADS)
    b = O.screen_rows(O.round_half(feats), O.half_ensemble(v), O.half_ensemble(p), w.thr, threads=THREADS)
    for x, y in zip(a[:3], b[:3]):
        assert np.array_equal(np.asarray(x), np.asarray(y))
