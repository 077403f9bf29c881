"""ctypes wrapper around the plain C oracle (``mlt_oracle.c``).

Test infrastructure only: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` use it.  The C file is compiled with gcc
(``-ffp-contract=off``: no fused multiply-add) into ``oracle/_build``.

Every function takes plain numpy arrays.  An ensemble is anything with
``nodes`` (structured array, 12-byte heap-order slots), ``n_trees`` and
``depth`` attributes, or a ``(nodes, n_trees, depth)`` tuple.
"""
from __future__ import annotations

import concurrent.futures as _cf
import ctypes as C
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mlt_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "libmlt_oracle.so")

# Documented input layouts (ML^2Tuner screening interface).
NODE_DTYPE = np.dtype(
    [("feature", "<i4"), ("value", "<f4"), ("default_left", "u1"), ("pad", "u1", (3,))]
)
OP_DTYPE = np.dtype([("op", "<i4"), ("a", "<i4"), ("b", "<i4"), ("c", "<f4")])

_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile the oracle shared library (idempotent); return its path."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    stale = (
        not os.path.exists(_LIB_PATH)
        or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    )
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = [
            "gcc", "-O2", "-std=c99", "-ffp-contract=off", "-fno-fast-math",
            "-fPIC", "-shared", "-o", tmp, _SRC, "-lm",
        ]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = C.CDLL(build())
        P = C.c_void_p
        i64, i32, f32 = C.c_int64, C.c_int, C.c_float
        lib.orc_tree_leaf.argtypes = [P, i32, P]
        lib.orc_tree_leaf.restype = f32
        lib.orc_margins.argtypes = [P, i32, i32, P, i64, i32, P]
        lib.orc_margins.restype = None
        lib.orc_tau.argtypes = [f32]
        lib.orc_tau.restype = f32
        lib.orc_sigmoid.argtypes = [f32]
        lib.orc_sigmoid.restype = f32
        lib.orc_screen_rows.argtypes = [P, i64, i32, P, i32, i32, P, i32, i32, f32, P, P, P, P]
        lib.orc_screen_rows.restype = i32
        lib.orc_topk.argtypes = [P, P, i64, i32, i64, P]
        lib.orc_topk.restype = i64
        lib.orc_screen.argtypes = [P, i64, i32, P, i32, i32, P, i32, i32, f32, i32, P, P, P]
        lib.orc_screen.restype = i64
        lib.orc_rerank.argtypes = [P, i32, P, i64, P, i32, i32, i32, P, P]
        lib.orc_rerank.restype = i64
        lib.orc_sa_step.argtypes = [P, P, i32, P, i32, P, i32, i32, P, i32, i32, P, P, P, P, P, i64, f32, f32,
                                    P, P, P]
        lib.orc_sa_step.restype = i32
        lib.orc_decode.argtypes = [P, i32, i64, i64, P]
        lib.orc_decode.restype = i32
        lib.orc_features.argtypes = [P, P, i32, P, i32, i64, i64, P, P]
        lib.orc_features.restype = i32
        _lib = lib
        return lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def _ens(e):
    if isinstance(e, tuple):
        nodes, n_trees, depth = e
    else:
        nodes, n_trees, depth = e.nodes, e.n_trees, e.depth
    nodes = np.ascontiguousarray(nodes)
    if nodes.dtype.itemsize != 12:
        raise ValueError("node slots must be 12 bytes")
    slots = (2 << depth) - 1
    if nodes.size != n_trees * slots:
        raise ValueError("node array size does not match n_trees and depth")
    return nodes, int(n_trees), int(depth)


def _f32_2d(feats):
    feats = np.ascontiguousarray(feats, dtype=np.float32)
    if feats.ndim != 2:
        raise ValueError("features must be [n][F]")
    return feats


def _chunks(n, threads):
    threads = max(1, min(int(threads), n if n > 0 else 1))
    edges = np.linspace(0, n, threads + 1).astype(np.int64)
    return [(int(a), int(b)) for a, b in zip(edges[:-1], edges[1:]) if b > a]


def tree_leaf(tree_nodes, depth: int, x) -> float:
    """Leaf value one tree routes the feature vector x to."""
    lib = _load()
    t = np.ascontiguousarray(tree_nodes)
    xv = np.ascontiguousarray(x, dtype=np.float32)
    return float(lib.orc_tree_leaf(_ptr(t), int(depth), _ptr(xv)))


def margins(ensemble, feats, threads: int = 1) -> np.ndarray:
    """Ensemble margin (sum of leaves, fp32, tree order) for every row.

    Rows are independent, so ``threads`` > 1 splits them over host threads
    (ctypes releases the GIL); every row is still computed by the same
    single-threaded routine, so the result does not depend on the split.
    """
    lib = _load()
    nodes, n_trees, depth = _ens(ensemble)
    feats = _f32_2d(feats)
    n, F = feats.shape
    out = np.empty(n, dtype=np.float32)

    def run(a, b):
        lib.orc_margins(_ptr(nodes), n_trees, depth, feats[a:].ctypes.data, b - a, F,
                        out[a:].ctypes.data)

    parts = _chunks(n, threads)
    if len(parts) <= 1:
        for a, b in parts:
            run(a, b)
    else:
        with _cf.ThreadPoolExecutor(len(parts)) as ex:
            list(ex.map(lambda ab: run(*ab), parts))
    return out


def tau(thr: float) -> float:
    """Smallest float margin m with sigmoid(m) >= thr (NaN if thr not in (0,1))."""
    return float(_load().orc_tau(float(thr)))


def sigmoid(m: float) -> float:
    return float(_load().orc_sigmoid(float(m)))


def screen_rows(feats, v_ens, p_ens, thr: float, threads: int = 1):
    """Per-row screening: (pvalid, perf, valid, margin_v) for every row."""
    lib = _load()
    vn, vt, vd = _ens(v_ens)
    pn, pt, pd = _ens(p_ens)
    feats = _f32_2d(feats)
    n, F = feats.shape
    pvalid = np.empty(n, np.float32)
    perf = np.empty(n, np.float32)
    valid = np.empty(n, np.uint8)
    mv = np.empty(n, np.float32)
    status = []

    def run(a, b):
        status.append(lib.orc_screen_rows(
            feats[a:].ctypes.data, b - a, F, _ptr(vn), vt, vd, _ptr(pn), pt, pd,
            float(thr), pvalid[a:].ctypes.data, perf[a:].ctypes.data,
            valid[a:].ctypes.data, mv[a:].ctypes.data))

    parts = _chunks(n, threads)
    if len(parts) <= 1:
        for a, b in parts:
            run(a, b)
    else:
        with _cf.ThreadPoolExecutor(len(parts)) as ex:
            list(ex.map(lambda ab: run(*ab), parts))
    if any(s != 0 for s in status):
        raise ValueError("threshold must lie in (0, 1)")
    return pvalid, perf, valid.astype(bool), mv


def topk(perf, valid, k: int, index_base: int = 0):
    """(top-k indices padded with -1, survivor count) by a full sort."""
    lib = _load()
    perf = np.ascontiguousarray(perf, dtype=np.float32)
    valid_u8 = np.ascontiguousarray(valid, dtype=np.uint8)
    out = np.empty(int(k), dtype=np.int64)
    s = lib.orc_topk(_ptr(perf), _ptr(valid_u8), perf.size, int(k), int(index_base), _ptr(out))
    if s < 0:
        raise MemoryError("oracle top-k allocation failed")
    return out, int(s)


def screen(feats, v_ens, p_ens, thr: float, k: int):
    """Whole pass, single-threaded: (pvalid, perf, topk, survivor count)."""
    lib = _load()
    vn, vt, vd = _ens(v_ens)
    pn, pt, pd = _ens(p_ens)
    feats = _f32_2d(feats)
    n, F = feats.shape
    pvalid = np.empty(n, np.float32)
    perf = np.empty(n, np.float32)
    out = np.empty(int(k), np.int64)
    s = lib.orc_screen(_ptr(feats), n, F, _ptr(vn), vt, vd, _ptr(pn), pt, pd,
                       float(thr), int(k), _ptr(pvalid), _ptr(perf), _ptr(out))
    if s < 0:
        raise ValueError("oracle screen failed (threshold outside (0,1) or no memory)")
    return pvalid, perf, out, int(s)


def rerank(feats, cand, a_ens, n_final: int):
    """Model A rerank of the kept candidates: (scores [m], final [n_final])."""
    lib = _load()
    an, at, ad = _ens(a_ens)
    feats = _f32_2d(feats)
    cand = np.ascontiguousarray(cand, dtype=np.int64)
    score = np.empty(cand.size, np.float32)
    final = np.empty(int(n_final), np.int64)
    v = lib.orc_rerank(_ptr(feats), feats.shape[1], _ptr(cand), cand.size, _ptr(an), at, ad,
                       int(n_final), _ptr(score), _ptr(final))
    if v < 0:
        raise MemoryError("oracle rerank allocation failed")
    return score, final


def sa_step(radices, option_values, program, v_ens, p_ens, parent, parent_score, knob_draw, digit_draw,
            log_u, temperature: float, thr: float):
    """One explorer proposal step: (next [m] int64, next_score [m] f32, accepted [m] i32)."""
    lib = _load()
    r = np.ascontiguousarray(radices, dtype=np.int32)
    ov = np.ascontiguousarray(option_values, dtype=np.float32)
    prog = np.ascontiguousarray(program)
    vn, vt, vd = _ens(v_ens)
    pn, pt, pd = _ens(p_ens)
    parent = np.ascontiguousarray(parent, dtype=np.int64)
    ps = np.ascontiguousarray(parent_score, dtype=np.float32)
    kd = np.ascontiguousarray(knob_draw, dtype=np.uint32)
    dd = np.ascontiguousarray(digit_draw, dtype=np.uint32)
    lu = np.ascontiguousarray(log_u, dtype=np.float32)
    m = parent.size
    nxt = np.empty(m, np.int64)
    nsc = np.empty(m, np.float32)
    acc = np.empty(m, np.int32)
    rc = lib.orc_sa_step(_ptr(r), _ptr(ov), r.size, _ptr(prog), prog.size, _ptr(vn), vt, vd, _ptr(pn), pt, pd,
                         _ptr(parent), _ptr(ps), _ptr(kd), _ptr(dd), _ptr(lu), m, float(temperature), float(thr),
                         _ptr(nxt), _ptr(nsc), _ptr(acc))
    if rc != 0:
        raise ValueError("malformed program or threshold")
    return nxt, nsc, acc


def decode(radices, first: int, n: int) -> np.ndarray:
    """[n][n_knobs] option indices of candidates first .. first+n-1."""
    lib = _load()
    r = np.ascontiguousarray(radices, dtype=np.int32)
    out = np.empty((int(n), r.size), dtype=np.uint8)
    if lib.orc_decode(_ptr(r), r.size, int(first), int(n), _ptr(out)) != 0:
        raise ValueError("candidate index beyond the knob space")
    return out


def features(radices, option_values, program, first: int, n: int, threads: int = 1):
    """(knobs [n][n_knobs] u8, feats [n][F] f32) for candidates first .. first+n-1."""
    lib = _load()
    r = np.ascontiguousarray(radices, dtype=np.int32)
    ov = np.ascontiguousarray(option_values, dtype=np.float32)
    prog = np.ascontiguousarray(program)
    if prog.dtype.itemsize != 16:
        raise ValueError("feature ops must be 16 bytes")
    F = prog.size
    knobs = np.empty((int(n), r.size), dtype=np.uint8)
    feats = np.empty((int(n), F), dtype=np.float32)
    status = []

    def run(a, b):
        status.append(lib.orc_features(_ptr(r), _ptr(ov), r.size, _ptr(prog), F,
                                       int(first) + a, b - a, knobs[a:].ctypes.data,
                                       feats[a:].ctypes.data))

    parts = _chunks(int(n), threads)
    if len(parts) <= 1:
        for a, b in parts:
            run(a, b)
    else:
        with _cf.ThreadPoolExecutor(len(parts)) as ex:
            list(ex.map(lambda ab: run(*ab), parts))
    if any(s != 0 for s in status):
        raise ValueError("index beyond the knob space or malformed feature program")
    return knobs, feats


# ---------------------------------------------------------------------------
# Half tables (binary16 thresholds, leaves and features): the rounded model
# ---------------------------------------------------------------------------
def round_half(a) -> np.ndarray:
    """IEEE 754 binary16 rounding of fp32 values (round to nearest, ties to
    even; magnitudes from 65520 up become infinities; NaN stays NaN),
    returned as fp32 -- exact, since every binary16 value is an fp32 value.
    numpy's float16 conversion implements this rounding."""
    with np.errstate(over="ignore"):
        return np.asarray(a, dtype=np.float32).astype(np.float16).astype(np.float32)


def half_ensemble(ensemble):
    """The ensemble half tables hold: every split threshold and leaf value
    rounded to binary16 (same shape and features).  Screening the rounded
    rows (round_half) with it is the half-table variant's exact result."""
    nodes, n_trees, depth = _ens(ensemble)
    out = np.array(nodes, copy=True)
    used = out["feature"] != -2
    out["value"][used] = round_half(out["value"][used])
    return (out, n_trees, depth)

