"""Python binding of libmlt (ctypes): argument marshalling only.

Every step of screening runs in the CUDA library; this module only turns
torch tensors / numpy arrays into pointers and sizes, passes the current
CUDA stream, and raises MltError on a non-zero status.  There is no CPU
fallback: if libmlt.so cannot be built or loaded, the calls raise.
"""
from __future__ import annotations

import ctypes as C
import os
import re
import threading

import numpy as np

from . import _build

MLT_MODEL_V, MLT_MODEL_P, MLT_MODEL_A = 0, 1, 2
STATUS = {0: "MLT_OK", -1: "MLT_EINVAL", -2: "MLT_ENOMODEL", -3: "MLT_ECUDA", -4: "MLT_ENOMEM",
          -5: "MLT_ETIMEOUT"}

NODE_DTYPE = np.dtype(
    [("feature", "<i4"), ("value", "<f4"), ("default_left", "u1"), ("pad", "u1", (3,))]
)
OP_DTYPE = np.dtype([("op", "<i4"), ("a", "<i4"), ("b", "<i4"), ("c", "<f4")])

HEADER = os.path.join(_build.ROOT, "include", "mlt.h")


class MltError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"{STATUS.get(code, code)}: {message}")
        self.code = code


_lib = None
_lock = threading.Lock()


def library_path() -> str:
    return _build.LIB_PATH


def lib(build_if_missing: bool = True):
    """Load libmlt.so (building it first when missing or stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if build_if_missing:
            _build.build()
        if not os.path.exists(_build.LIB_PATH):
            raise RuntimeError(f"libmlt.so missing at {_build.LIB_PATH}")
        L = C.CDLL(_build.LIB_PATH)
        P, i32, i64, f32 = C.c_void_p, C.c_int, C.c_int64, C.c_float
        sig = {
            "mlt_set_num_features": [i32],
            "mlt_load_ensemble": [i32, P, i32, i32],
            "mlt_load_ensemble_f16": [i32, P, i32, i32],
            "mlt_screen_host_batches": [P, i64, P, i64, f32, i32, P, P, P],
            "mlt_selftest_wait_timeout": [P, i64],
            "mlt_selftest_walk_timeout": [i32, i64],
            "mlt_selftest_poison_state": [i32, C.c_uint32],
            "mlt_free_ensemble": [i32],
            "mlt_validity_cut": [f32, P],
            "mlt_screen": [P, P, i64, f32, i32, P, P, P],
            "mlt_screen_host": [P, P, i64, f32, i32, P, P, P],
            "mlt_decode_knobs": [P, P, P, i32, P, i32, i64, i64, P, P],
            "mlt_screen_decoded": [P, P, P, i32, P, i64, i64, f32, i32, P, P, P],
            "mlt_sync_status": [P],
            "mlt_last_survivor_count": [P, P],
            "mlt_profile_phases": [i32],
            "mlt_phase_times": [P, i32, P],
            "mlt_tune_walk": [i32, i32, i32, i32, i32, i32],
            "mlt_walk_shape": [i32, i64, i32, P],
            "mlt_tune_head_levels": [i32],
            "mlt_tune_fused_small": [i32],
            "mlt_tune_decode_jit": [i64],
            "mlt_decode_jit_available": [],
            "mlt_walk_peak": [P, i32, P, i64, i32, P, P],
            "mlt_screen_noalloc": [P, P, i64, f32, i32, P, P, P],
            "mlt_rerank": [P, P, i64, P, i32, i32, P, P],
            "mlt_merge_topk": [P, P, P, i64, i32, P],
            "mlt_screen_until": [P, P, i64, i64, i64, f32, i32, P, P, P, P],
            "mlt_screen_until_decoded": [P, P, P, i32, P, i64, i64, i64, i64, f32, i32, P, P, P, P],
            "mlt_sa_step": [P, P, P, i32, P, P, P, P, P, P, i64, f32, f32, P, P, P],
        }
        for name, args in sig.items():
            fn = getattr(L, name)
            fn.argtypes = args
            fn.restype = i32
        L.mlt_kernel_launches.argtypes = []
        L.mlt_kernel_launches.restype = i64
        L.mlt_decode_jit_calls.argtypes = []
        L.mlt_decode_jit_calls.restype = i64
        L.mlt_last_error.argtypes = []
        L.mlt_last_error.restype = C.c_char_p
        _lib = L
        return L


def declared_symbols() -> list[str]:
    """Every function the C header declares."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(mlt_\w+)\s*\(", text, re.M)))


def _check(rc: int):
    if rc != 0:
        msg = lib().mlt_last_error()
        raise MltError(rc, msg.decode() if msg else "")


def _stream_ptr(stream=None):
    import torch

    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def _dptr(t):
    return C.c_void_p(0 if t is None else t.data_ptr())


# ---------------------------------------------------------------------------
# Model management
# ---------------------------------------------------------------------------

def set_num_features(F: int) -> None:
    _check(lib().mlt_set_num_features(int(F)))


def load_ensemble(model_id: int, nodes: np.ndarray, n_trees: int, depth: int) -> None:
    nodes = np.ascontiguousarray(nodes)
    if nodes.dtype.itemsize != 12:
        raise ValueError("nodes must use the 12-byte slot layout")
    if nodes.size != n_trees * ((2 << depth) - 1):
        raise ValueError("node array size does not match n_trees and depth")
    _check(lib().mlt_load_ensemble(int(model_id), nodes.ctypes.data, int(n_trees), int(depth)))


def load_ensemble_f16(model_id: int, nodes: np.ndarray, n_trees: int, depth: int) -> None:
    """Load model V or P as half tables (binary16 thresholds, leaves and
    staged features: changes results, see mlt_load_ensemble_f16)."""
    nodes = np.ascontiguousarray(nodes)
    if nodes.dtype.itemsize != 12:
        raise ValueError("nodes must use the 12-byte slot layout")
    if nodes.size != n_trees * ((2 << depth) - 1):
        raise ValueError("node array size does not match n_trees and depth")
    _check(lib().mlt_load_ensemble_f16(int(model_id), nodes.ctypes.data, int(n_trees), int(depth)))


def free_ensemble(model_id: int) -> None:
    _check(lib().mlt_free_ensemble(int(model_id)))


def validity_cut(thr: float) -> float:
    out = C.c_float()
    _check(lib().mlt_validity_cut(C.c_float(thr), C.byref(out)))
    return out.value


# ---------------------------------------------------------------------------
# Screening
# ---------------------------------------------------------------------------

def _outputs(n, k, device, out_pvalid, out_perf, out_topk):
    import torch

    if out_pvalid is None:
        out_pvalid = torch.empty(n, dtype=torch.float32, device=device)
    if out_perf is None:
        out_perf = torch.empty(n, dtype=torch.float32, device=device)
    if out_topk is None:
        out_topk = torch.empty(k, dtype=torch.int64, device=device)
    return out_pvalid, out_perf, out_topk


def screen(feats, thr: float, k: int, out_pvalid=None, out_perf=None, out_topk=None, stream=None):
    """Screen a [n][F] fp32 CUDA tensor: returns (pvalid, perf, topk) tensors."""
    import torch

    if not (isinstance(feats, torch.Tensor) and feats.is_cuda and feats.dtype == torch.float32):
        raise TypeError("feats must be a float32 CUDA tensor")
    if not feats.is_contiguous() or feats.dim() != 2:
        raise ValueError("feats must be a contiguous [n][F] tensor")
    n = feats.shape[0]
    pv, pf, tk = _outputs(n, k, feats.device, out_pvalid, out_perf, out_topk)
    _check(lib().mlt_screen(_stream_ptr(stream), _dptr(feats), n, C.c_float(thr), int(k),
                            _dptr(pv), _dptr(pf), _dptr(tk)))
    return pv, pf, tk


def screen_noalloc(feats, thr: float, k: int, out_pvalid=None, out_perf=None, out_topk=None,
                   stream=None):
    """mlt_screen_noalloc: like screen(), with the library's fixed scratch
    (n <= 262,144; overlapping calls race)."""
    import torch

    if not (isinstance(feats, torch.Tensor) and feats.is_cuda and feats.dtype == torch.float32):
        raise TypeError("feats must be a float32 CUDA tensor")
    n = feats.shape[0]
    pv, pf, tk = _outputs(n, k, feats.device, out_pvalid, out_perf, out_topk)
    _check(lib().mlt_screen_noalloc(_stream_ptr(stream), _dptr(feats), n, C.c_float(thr), int(k),
                                    _dptr(pv), _dptr(pf), _dptr(tk)))
    return pv, pf, tk


def screen_until(feats, batch: int, target: int, thr: float, k: int, with_outputs=True, stream=None):
    """Batched accumulation over the rows of `feats`: returns (pvalid, perf,
    topk, stats) with stats = [consumed, kept, batches] (CUDA tensors)."""
    import torch

    n = feats.shape[0]
    pv = torch.empty(n, dtype=torch.float32, device=feats.device) if with_outputs else None
    pf = torch.empty(n, dtype=torch.float32, device=feats.device) if with_outputs else None
    tk = torch.empty(int(k), dtype=torch.int64, device=feats.device)
    stats = torch.empty(3, dtype=torch.int64, device=feats.device)
    _check(lib().mlt_screen_until(_stream_ptr(stream), _dptr(feats), n, int(batch), int(target), C.c_float(thr),
                                  int(k), _dptr(pv), _dptr(pf), _dptr(tk), _dptr(stats)))
    return pv, pf, tk, stats


def screen_until_decoded(radices, option_values, program, first_index: int, n_total: int, batch: int,
                         target: int, thr: float, k: int, device="cuda", with_outputs=True, stream=None):
    """Batched accumulation over a decoded knob space."""
    import torch

    r, ov, prog = _decoder_args(radices, option_values, program)
    pv = torch.empty(n_total, dtype=torch.float32, device=device) if with_outputs else None
    pf = torch.empty(n_total, dtype=torch.float32, device=device) if with_outputs else None
    tk = torch.empty(int(k), dtype=torch.int64, device=device)
    stats = torch.empty(3, dtype=torch.int64, device=device)
    _check(lib().mlt_screen_until_decoded(_stream_ptr(stream), r.ctypes.data, ov.ctypes.data, r.size,
                                          prog.ctypes.data, int(first_index), int(n_total), int(batch),
                                          int(target), C.c_float(thr), int(k), _dptr(pv), _dptr(pf),
                                          _dptr(tk), _dptr(stats)))
    return pv, pf, tk, stats


def sa_step(radices, option_values, program, parent, parent_score, knob_draw, digit_draw, log_u,
            temperature: float, thr: float, stream=None):
    """One explorer proposal step over the chains in `parent` (CUDA tensors:
    int64, float32, uint32-as-int32, int32, float32): returns (next,
    next_score, accepted) CUDA tensors."""
    import torch

    r, ov, prog = _decoder_args(radices, option_values, program)
    m = parent.numel()
    nxt = torch.empty(m, dtype=torch.int64, device=parent.device)
    nsc = torch.empty(m, dtype=torch.float32, device=parent.device)
    acc = torch.empty(m, dtype=torch.int32, device=parent.device)
    _check(lib().mlt_sa_step(_stream_ptr(stream), r.ctypes.data, ov.ctypes.data, r.size, prog.ctypes.data,
                             _dptr(parent), _dptr(parent_score), _dptr(knob_draw), _dptr(digit_draw), _dptr(log_u),
                             m, C.c_float(temperature), C.c_float(thr), _dptr(nxt), _dptr(nsc), _dptr(acc)))
    return nxt, nsc, acc


def rerank(feats, cand, n_final: int, out_score=None, out_final=None, stream=None):
    """Model A's rerank of candidate indices `cand` (CUDA int64 tensor) whose
    rows are in `feats`: returns (scores [m], final [n_final])."""
    import torch

    if not (isinstance(cand, torch.Tensor) and cand.is_cuda and cand.dtype == torch.int64):
        raise TypeError("cand must be an int64 CUDA tensor")
    m = cand.numel()
    if out_score is None:
        out_score = torch.empty(m, dtype=torch.float32, device=cand.device)
    if out_final is None:
        out_final = torch.empty(int(n_final), dtype=torch.int64, device=cand.device)
    _check(lib().mlt_rerank(_stream_ptr(stream), _dptr(feats), feats.shape[0], _dptr(cand), m, int(n_final),
                            _dptr(out_score), _dptr(out_final)))
    return out_score, out_final


def merge_topk(scores, indices, k: int, out=None, stream=None):
    """mlt_merge_topk: the k best (score, global index) pairs (CUDA fp32 and
    int64 tensors of equal length; a negative index is an empty slot) by
    (score desc, index asc), -1 padded: returns a CUDA int64 tensor [k]."""
    import torch

    for t, dt in ((scores, torch.float32), (indices, torch.int64)):
        if not (isinstance(t, torch.Tensor) and t.is_cuda and t.dtype == dt and t.is_contiguous()):
            raise TypeError("scores / indices must be contiguous float32 / int64 CUDA tensors")
    m = indices.numel()
    if scores.numel() != m:
        raise ValueError("scores and indices differ in length")
    if out is None:
        out = torch.empty(int(k), dtype=torch.int64, device=indices.device)
    _check(lib().mlt_merge_topk(_stream_ptr(stream), _dptr(scores), _dptr(indices), m, int(k), _dptr(out)))
    return out


def screen_host(feats: np.ndarray, thr: float, k: int, out=None, stream=None):
    """Screen a host [n][F] float32 array (copies in and out inside the call).

    `out` may be a (pvalid, perf, topk) triple of host arrays (for example
    pinned torch tensors' numpy views) to fill in place."""
    feats = np.ascontiguousarray(feats, dtype=np.float32)
    n = feats.shape[0]
    if out is None:
        out = (np.empty(n, np.float32), np.empty(n, np.float32), np.empty(k, np.int64))
    pv, pf, tk = out
    _check(lib().mlt_screen_host(_stream_ptr(stream), feats.ctypes.data, n, C.c_float(thr), int(k),
                                 pv.ctypes.data, pf.ctypes.data, tk.ctypes.data))
    return pv, pf, tk


def screen_host_batches(feats, thr: float, k: int, outs=None, stream=None):
    """Screen a list of host batches (each [n][F] fp32, page-locked for
    overlap) with the pipelined host entry point.  `outs`: a list of
    (pvalid, perf, topk) host arrays per batch (pvalid / perf may be None);
    allocated if omitted.  Returns the list."""
    feats = [np.asarray(f) for f in feats]
    nb = len(feats)
    n = feats[0].shape[0] if nb else 0
    for f in feats:
        if f.dtype != np.float32 or not f.flags.c_contiguous or f.shape[0] != n:
            raise ValueError("batches must be C-contiguous fp32 arrays of equal length")
    if outs is None:
        outs = [(np.empty(n, np.float32), np.empty(n, np.float32), np.empty(k, np.int64)) for _ in range(nb)]
    arr = lambda xs: (C.c_void_p * max(1, nb))(*[None if x is None else x.ctypes.data for x in xs])
    fp = arr(feats)
    pv = arr([o[0] for o in outs])
    pf = arr([o[1] for o in outs])
    tk = arr([o[2] for o in outs])
    _check(lib().mlt_screen_host_batches(_stream_ptr(stream), nb, fp, int(n), C.c_float(thr), int(k), pv, pf, tk))
    return outs


def _decoder_args(radices, option_values, program):
    r = np.ascontiguousarray(radices, dtype=np.int32)
    ov = np.ascontiguousarray(option_values, dtype=np.float32)
    prog = np.ascontiguousarray(program)
    if prog.dtype.itemsize != 16:
        raise ValueError("program must use the 16-byte op layout")
    return r, ov, prog


def decode_knobs(radices, option_values, program, first_index: int, n: int, device="cuda",
                 want_knobs=True, want_feats=True, stream=None):
    """(knobs [n][K] uint8, feats [n][F] fp32) CUDA tensors (None if not wanted)."""
    import torch

    r, ov, prog = _decoder_args(radices, option_values, program)
    knobs = torch.empty((n, r.size), dtype=torch.uint8, device=device) if want_knobs else None
    feats = torch.empty((n, prog.size), dtype=torch.float32, device=device) if want_feats else None
    _check(lib().mlt_decode_knobs(_stream_ptr(stream), r.ctypes.data, ov.ctypes.data, r.size,
                                  prog.ctypes.data, prog.size, int(first_index), int(n),
                                  _dptr(knobs), _dptr(feats)))
    return knobs, feats


def screen_decoded(radices, option_values, program, first_index: int, n: int, thr: float, k: int,
                   device="cuda", out_pvalid=None, out_perf=None, out_topk=None, stream=None):
    """Screen candidates first_index .. first_index+n-1 of a knob space."""
    r, ov, prog = _decoder_args(radices, option_values, program)
    pv, pf, tk = _outputs(n, k, device, out_pvalid, out_perf, out_topk)
    _check(lib().mlt_screen_decoded(_stream_ptr(stream), r.ctypes.data, ov.ctypes.data, r.size,
                                    prog.ctypes.data, int(first_index), int(n), C.c_float(thr),
                                    int(k), _dptr(pv), _dptr(pf), _dptr(tk)))
    return pv, pf, tk


def sync_status(stream=None) -> None:
    _check(lib().mlt_sync_status(_stream_ptr(stream)))


def selftest_wait_timeout(limit_ns: int, stream=None) -> None:
    """Launch the failure-detection self-test (a device wait that runs out);
    the next sync_status raises MltError with MLT_ETIMEOUT."""
    _check(lib().mlt_selftest_wait_timeout(_stream_ptr(stream), int(limit_ns)))


def selftest_walk_timeout(cta: int, limit_ns: int) -> None:
    """Arm the in-path self-test: the next screening call's V pass (full
    table) makes CTA `cta` give up waiting for its first tree chunk after
    limit_ns; the next sync_status raises MltError with MLT_ETIMEOUT."""
    _check(lib().mlt_selftest_walk_timeout(int(cta), int(limit_ns)))


def selftest_poison_state(value: int, static_scratch: bool = False) -> None:
    """Write `value` into the selection state's counters (as a call that
    stopped part-way could leave them); the next call must not notice."""
    _check(lib().mlt_selftest_poison_state(1 if static_scratch else 0, C.c_uint32(value)))


def walk_peak(feats, rounds: int, model_id: int = MLT_MODEL_V, out_sums=None, stream=None):
    """mlt_walk_peak: walk the first trees of a full-table model, held in
    shared memory, `rounds` times for every row of `feats` (a [n][F] fp32
    CUDA tensor).  Returns (sums, visits): the per-row fp32 leaf sums and the
    node visits of the launch (time it with events on `stream`)."""
    import torch

    if not (isinstance(feats, torch.Tensor) and feats.is_cuda and feats.dtype == torch.float32):
        raise TypeError("feats must be a float32 CUDA tensor")
    if not feats.is_contiguous() or feats.dim() != 2:
        raise ValueError("feats must be a contiguous [n][F] tensor")
    n = feats.shape[0]
    if out_sums is None:
        out_sums = torch.empty(n, dtype=torch.float32, device=feats.device)
    visits = C.c_int64()
    _check(lib().mlt_walk_peak(_stream_ptr(stream), int(model_id), _dptr(feats), n, int(rounds), _dptr(out_sums),
                               C.byref(visits)))
    return out_sums, int(visits.value)


def last_survivor_count(stream=None) -> int:
    out = C.c_int64()
    _check(lib().mlt_last_survivor_count(_stream_ptr(stream), C.byref(out)))
    return int(out.value)


PHASES = ("v_pass", "compaction", "p_pass", "topk")


def profile_phases(enable: bool) -> None:
    _check(lib().mlt_profile_phases(1 if enable else 0))


def phase_times():
    """({phase: summed ms}, recorded calls) since profiling was enabled."""
    out = (C.c_float * 4)()
    calls = C.c_int64()
    _check(lib().mlt_phase_times(out, 4, C.byref(calls)))
    return dict(zip(PHASES, [float(v) for v in out])), int(calls.value)


def tune_walk(model_id: int, candidates: int = 0, splits: int = 0, group: int = 0, chunk_trees: int = 0,
              nbuf: int = 0) -> None:
    """Fix (or with zeros, release) the tree walk's launch shape for one model."""
    _check(lib().mlt_tune_walk(int(model_id), int(candidates), int(splits), int(group), int(chunk_trees),
                               int(nbuf)))


def tune_fused_small(max_n: int) -> None:
    """Batches up to max_n candidates (0 .. 8192) screen in one launch when
    their models allow it; 0 turns the single-launch path off."""
    _check(lib().mlt_tune_fused_small(int(max_n)))


def walk_shape(model_id: int, n: int, p_pass: bool = False) -> dict:
    """The launch shape the walk over model_id's trees would use for a
    screening call of n candidates (P pass: planned for about n/2)."""
    out = np.zeros(7, dtype=np.int32)
    _check(lib().mlt_walk_shape(int(model_id), int(n), 1 if p_pass else 0, out.ctypes.data))
    kinds = {0: "full", 1: "compact", 2: "half", 3: "split"}
    return {"candidates": int(out[0]), "splits": int(out[1]), "group": int(out[2]), "chunk_trees": int(out[3]),
            "nbuf": int(out[4]), "resident": int(out[5]), "table": kinds.get(int(out[6]), str(int(out[6])))}


def tune_decode_jit(min_n: int) -> None:
    """Decoded batches of at least min_n candidates build their rows with
    the feature program compiled at run time (NVRTC) and screen those; 0
    keeps every decoded batch on the interpreted in-walk path."""
    _check(lib().mlt_tune_decode_jit(int(min_n)))


def decode_jit_available() -> bool:
    """Whether NVRTC and the CUDA driver library load in this process."""
    return bool(lib().mlt_decode_jit_available())


def decode_jit_calls() -> int:
    """Screening calls so far that ran the compiled feature program."""
    return int(lib().mlt_decode_jit_calls())


def tune_head_levels(levels: int) -> None:
    """Table format of deep (depth > 10) V and P models loaded afterwards:
    6 or 7 head levels in shared memory (split table), or 0 (compact)."""
    _check(lib().mlt_tune_head_levels(int(levels)))


def kernel_launches() -> int:
    return int(lib().mlt_kernel_launches())


def load_workload_models(w, half: bool = False) -> None:
    """Set F and load the workload's V and P ensembles (as half tables if
    `half`)."""
    set_num_features(w.cfg.F if w.feats is None else w.feats.shape[1])
    load = load_ensemble_f16 if half else load_ensemble
    load(MLT_MODEL_V, w.v.nodes, w.v.n_trees, w.v.depth)
    load(MLT_MODEL_P, w.p.nodes, w.p.n_trees, w.p.depth)
