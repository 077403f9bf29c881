"""Shared helpers of the GPU parity tests: run a workload through the CUDA
library and through the oracle on the same seeded inputs."""
import os

import numpy as np

import oracle as O
from paper_2411_10764_gb300 import mlt

# the oracle's rows are independent: split them over every host core
THREADS = max(1, os.cpu_count() or 1)


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


def oracle_screen_chunked(w, thr=None, k=None, chunk=1 << 20):
    """The oracle's screening of the whole workload, `chunk` rows at a time
    (a decoded workload is decoded by the oracle chunk by chunk, so its
    feature matrix is never held whole), every chunk split over all host
    cores; then one full sort for the top-k.  Returns (pvalid, perf, top-k,
    survivors, margin_v)."""
    thr = w.thr if thr is None else thr
    k = w.k if k is None else k
    n = w.n
    pv = np.empty(n, np.float32)
    pf = np.empty(n, np.float32)
    valid = np.empty(n, bool)
    mv = np.empty(n, np.float32)
    for a in range(0, n, chunk):
        b = min(n, a + chunk)
        if w.decoder is None:
            x = w.feats[a:b]
        else:
            d = w.decoder
            _, x = O.features(d.radices, d.option_values, d.program, w.first_index + a, b - a,
                              threads=THREADS)
        pv[a:b], pf[a:b], valid[a:b], mv[a:b] = O.screen_rows(x, w.v, w.p, thr, threads=THREADS)
    tk, s = O.topk(pf, valid, k, index_base=w.first_index)
    return pv, pf, tk, s, mv


def near_counts(margin_v, tau, perf, topk, index_base=0, rel=1e-6):
    """Candidates whose V margin lies within 1e-6 of the validity cut tau
    (absolute: tau is 0 at thr = 0.5) and survivors whose P score lies
    within 1e-6 (relative) of the k-th kept score."""
    near_tau = int(np.sum(np.abs(margin_v.astype(np.float64) - tau) <= rel * max(1.0, abs(tau))))
    kept = topk[topk >= 0] - index_base
    if kept.size == 0:
        return near_tau, 0
    kth = float(perf[kept[-1]])
    finite = perf[np.isfinite(perf)].astype(np.float64)
    near_k = int(np.sum(np.abs(finite - kth) <= rel * abs(kth)))
    return near_tau, near_k


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
