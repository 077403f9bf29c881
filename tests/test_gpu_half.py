"""GPU parity of the half-table variant: screening with binary16 tables
(mlt_load_ensemble_f16) equals the oracle's exact screening of the rounded
rows with the rounded model, bit for bit (decisions, survivor sets, P scores,
top-k); pvalid within 1e-6 relative.  Its distance from the fp32 model is
checked on the CPU (test_half_tables.py)."""
import dataclasses

import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_parity

pytestmark = pytest.mark.gpu


def gpu_half(w, feats=None, thr=None, k=None):
    import torch

    mlt.load_workload_models(w, half=True)
    x = torch.from_numpy(w.feats if feats is None else feats).cuda()
    pv, pf, tk = mlt.screen(x, w.thr if thr is None else thr, w.k if k is None else k)
    mlt.sync_status()
    return pv.cpu().numpy(), pf.cpu().numpy(), tk.cpu().numpy(), mlt.last_survivor_count()


def oracle_half(w, feats=None, thr=None, k=None):
    x = O.round_half(w.feats if feats is None else feats)
    pv, pf, valid, _ = O.screen_rows(x, O.half_ensemble(w.v), O.half_ensemble(w.p),
                                     w.thr if thr is None else thr, threads=THREADS)
    tk, s = O.topk(pf, valid, w.k if k is None else k)
    return pv, pf, tk, s


@pytest.mark.parametrize("cid,n", [(1, 4096), (2, 20000), (3, 9001)])
def test_half_tables_match_rounded_oracle(cid, n):
    w = W.make_workload(cid, seed=1, n=n)
    assert_parity(gpu_half(w), oracle_half(w))


@pytest.mark.parametrize("n", [0, 1, 33, 257])
def test_half_tables_tiny_batches(n):
    w = W.make_workload(2, seed=4, n=max(n, 1))
    feats = w.feats[:n]
    got = gpu_half(w, feats=feats)
    exp = oracle_half(w, feats=feats)
    assert_parity(got, exp)


def test_half_tables_special_values():
    """NaN (both default sides), infinities, -0, magnitudes that overflow
    binary16, and values that round onto a threshold (ties)."""
    w = W.make_workload(2, seed=5, n=6000)
    x = w.feats.copy()
    rng = np.random.default_rng(3)
    rows = rng.choice(x.shape[0], 1500, replace=False)
    cols = rng.integers(0, x.shape[1], 1500)
    specials = np.array([np.nan, np.inf, -np.inf, -0.0, 70000.0, -65520.0, 65519.0], np.float32)
    x[rows[:700], cols[:700]] = specials[rng.integers(0, specials.size, 700)]
    # values within binary16 rounding of a split threshold of the same feature
    nodes = w.p.nodes
    split = nodes["feature"] >= 0
    thr = nodes["value"][split]
    feat = nodes["feature"][split]
    pick = rng.integers(0, thr.size, 800)
    eps = rng.choice([-1.0, 1.0], 800) * rng.choice([2.0 ** -12, 2.0 ** -13, 0.0], 800)
    x[rows[700:], feat[pick]] = (thr[pick] * (1.0 + eps)).astype(np.float32)
    assert_parity(gpu_half(w, feats=x), oracle_half(w, feats=x))


def test_half_tables_padded_unbalanced_trees():
    w = W.make_workload(2, seed=6, n=7000)
    th = W._QuantileThresholds(w.feats[:4096])
    v = W.make_ensemble(w.cfg, "V", th, 11, n_trees=90, depth=9, split_prob=0.7, shape="unbalanced")
    p = W.make_ensemble(w.cfg, "P", th, 12, n_trees=150, depth=10, split_prob=0.7, shape="unbalanced")
    w = dataclasses.replace(w, v=v, p=p)
    assert_parity(gpu_half(w), oracle_half(w))


@pytest.mark.parametrize("thr,k", [(0.05, 16384), (0.5, 1), (0.95, 300)])
def test_half_tables_thresholds_and_k(thr, k):
    w = W.make_workload(2, seed=7, n=9000)
    assert_parity(gpu_half(w, thr=thr, k=k), oracle_half(w, thr=thr, k=k))


def test_half_tables_with_one_model_in_fp32():
    """V in fp32, P as half tables: the V pass stages fp32 features, the P
    pass binary16 ones."""
    import torch

    w = W.make_workload(2, seed=8, n=8000)
    mlt.set_num_features(w.feats.shape[1])
    mlt.load_ensemble(mlt.MLT_MODEL_V, w.v.nodes, w.v.n_trees, w.v.depth)
    mlt.load_ensemble_f16(mlt.MLT_MODEL_P, w.p.nodes, w.p.n_trees, w.p.depth)
    pv, pf, tk = mlt.screen(torch.from_numpy(w.feats).cuda(), w.thr, w.k)
    mlt.sync_status()
    got = (pv.cpu().numpy(), pf.cpu().numpy(), tk.cpu().numpy(), mlt.last_survivor_count())
    opv, _, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    mp = O.margins(O.half_ensemble(w.p), O.round_half(w.feats), threads=THREADS)
    opf = np.where(valid, mp, -np.inf).astype(np.float32)
    otk, s = O.topk(opf, valid, w.k)
    assert_parity(got, (opv, opf, otk, s))


def test_half_tables_reject_decoded_screening():
    w = W.make_workload(4, seed=1, n=1000)
    mlt.load_workload_models(w, half=True)
    d = w.decoder
    with pytest.raises(mlt.MltError):
        mlt.screen_decoded(d.radices, d.option_values, d.program, 0, 1000, w.thr, w.k)
    mlt.load_workload_models(w)  # fp32 tables work again
    mlt.screen_decoded(d.radices, d.option_values, d.program, 0, 1000, w.thr, w.k)
    mlt.sync_status()


def test_half_tables_through_the_other_entry_points():
    """Half tables behind the batched accumulation, the pipelined host
    batches and the allocation-free entry point: each equals the rounded
    model's oracle."""
    import ctypes as C

    import torch

    w = W.make_workload(2, seed=11, n=12000)
    mlt.load_workload_models(w, half=True)
    x = O.round_half(w.feats)
    vh, ph = O.half_ensemble(w.v), O.half_ensemble(w.p)
    opv, opf, valid, _ = O.screen_rows(x, vh, ph, w.thr, threads=THREADS)
    otk, s = O.topk(opf, valid, w.k)
    # batched accumulation over the whole batch (target never reached)
    _, pf, tk, stats = mlt.screen_until(torch.from_numpy(w.feats).cuda(), 4096, 10 ** 9, w.thr, w.k)
    mlt.sync_status()
    assert stats.cpu().tolist()[0] == w.n
    assert np.array_equal(tk.cpu().numpy(), otk)
    assert np.array_equal(pf.cpu().numpy().view(np.uint32), opf.view(np.uint32))
    # pipelined host batches
    pinned = torch.from_numpy(w.feats).pin_memory().numpy()
    (pv_h, pf_h, tk_h), = mlt.screen_host_batches([pinned], w.thr, w.k)
    assert_parity((pv_h, pf_h, tk_h, s), (opv, opf, otk, s))
    # allocation-free entry point
    L = mlt.lib()
    dx = torch.from_numpy(w.feats).cuda()
    pv2 = torch.empty(w.n, device="cuda")
    pf2 = torch.empty(w.n, device="cuda")
    tk2 = torch.empty(w.k, dtype=torch.int64, device="cuda")
    st = torch.cuda.current_stream()
    rc = L.mlt_screen_noalloc(C.c_void_p(st.cuda_stream), C.c_void_p(dx.data_ptr()), C.c_int64(w.n), C.c_float(w.thr),
                              C.c_int(w.k), C.c_void_p(pv2.data_ptr()), C.c_void_p(pf2.data_ptr()),
                              C.c_void_p(tk2.data_ptr()))
    assert rc == 0
    mlt.sync_status()
    assert_parity((pv2.cpu().numpy(), pf2.cpu().numpy(), tk2.cpu().numpy(), s), (opv, opf, otk, s))
    mlt.load_workload_models(w)
