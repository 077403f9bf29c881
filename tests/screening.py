"""Shared helpers of the GPU parity tests: run a workload through the CUDA
library and through the oracle on the same seeded inputs."""
import os

import numpy as np

import oracle as O
from paper_2411_10764_gb300 import mlt

THREADS = max(1, min(32, os.cpu_count() or 1))


def gpu_screen(w, thr=None, k=None, feats=None):
    import torch

    thr = w.thr if thr is None else thr
    k = w.k if k is None else k
    mlt.load_workload_models(w)
    if w.decoder is not None:
        d = w.decoder
        pv, pf, tk = mlt.screen_decoded(d.radices, d.option_values, d.program, w.first_index, w.n,
                                        thr, k)
    else:
        x = torch.from_numpy(w.feats if feats is None else feats).cuda()
        pv, pf, tk = mlt.screen(x, thr, k)
    mlt.sync_status()
    s = mlt.last_survivor_count()
    return pv.cpu().numpy(), pf.cpu().numpy(), tk.cpu().numpy(), s


def oracle_feats(w, rows=None):
    """Feature rows for the oracle (decoded by the oracle for the decoded workload)."""
    if w.decoder is None:
        return w.feats if rows is None else w.feats[rows]
    d = w.decoder
    if rows is None:
        _, f = O.features(d.radices, d.option_values, d.program, w.first_index, w.n, threads=THREADS)
        return f
    out = np.empty((len(rows), d.program.size), np.float32)
    for i, r in enumerate(rows):
        _, f = O.features(d.radices, d.option_values, d.program, w.first_index + int(r), 1)
        out[i] = f[0]
    return out


def oracle_screen(w, thr=None, k=None, feats=None):
    thr = w.thr if thr is None else thr
    k = w.k if k is None else k
    x = oracle_feats(w) if feats is None else feats
    pv, pf, valid, _ = O.screen_rows(x, w.v, w.p, thr, threads=THREADS)
    tk, s = O.topk(pf, valid, k, index_base=w.first_index)
    return pv, pf, tk, s


def assert_same_bits(a, b, what, nan_equal=False):
    """Bit-for-bit equality of float32 arrays.  With nan_equal, a NaN matches
    any NaN: IEEE 754 leaves the bits of a NaN an operation generates to the
    implementation (the GPU gives 0x7FFFFFFF, an Arm host 0x7FC00000)."""
    a = np.asarray(a, np.float32).ravel()
    b = np.asarray(b, np.float32).ravel()
    diff = a.view(np.uint32) != b.view(np.uint32)
    if nan_equal:
        diff &= ~(np.isnan(a) & np.isnan(b))
    bad = np.nonzero(diff)[0]
    assert bad.size == 0, f"{what}: {bad.size} mismatches, first at {bad[:5]}: {a[bad[:5]]} vs {b[bad[:5]]}"


def assert_pvalid(g, o, rel=1e-6):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    err = np.abs(g - o) / np.maximum(np.abs(o), 1e-30)
    assert np.all(err <= rel), f"pvalid: max rel err {err.max():.3g} at {np.argmax(err)}"


def assert_parity(gpu, orc):
    gpv, gpf, gtk, gs = gpu
    opv, opf, otk, os_ = orc
    assert gs == os_, f"survivors {gs} vs {os_}"
    assert_same_bits(gpf, opf, "perf")
    assert_pvalid(gpv, opv)
    assert np.array_equal(gtk, otk), f"top-k differs: {gtk[:10]} vs {otk[:10]}"


def topk_from_scores(perf, k, index_base=0):
    """First k of the full order (score desc, index asc) over finite scores."""
    idx = np.nonzero(perf > -np.inf)[0]
    order = idx[np.lexsort((idx, -perf[idx].astype(np.float64)))]
    out = np.full(k, -1, np.int64)
    m = min(k, order.size)
    out[:m] = order[:m] + index_base
    return out, idx.size
