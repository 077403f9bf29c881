"""mlt_screen_noalloc against mlt_screen.

The no-allocation entry point serves callers that cannot call cudaMalloc
during a screening call (their device memory belongs to another allocator,
or cudaMalloc's implicit synchronisation is too costly in their loop).  It
runs the same kernels on a fixed scratch array inside the library, so its
outputs must equal those of the allocating entry point: P scores, survivor
set and top-k bit for bit, pvalid within the 1e-6 relative tolerance the
other parity tests use.  Two calls in a row check that the shared array's
leftover contents from one call do not leak into the next.

This file is collected last on purpose (a failure here leaves every other
test already run)."""
import ctypes as C

import numpy as np
import pytest

from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import assert_pvalid, assert_same_bits

pytestmark = pytest.mark.gpu


def _call(L, stream, x, n, thr, k, pv, pf, tk):
    return L.mlt_screen_noalloc(C.c_void_p(stream.cuda_stream), C.c_void_p(x.data_ptr()), C.c_int64(n),
                                C.c_float(thr), C.c_int(k), C.c_void_p(pv.data_ptr()),
                                C.c_void_p(pf.data_ptr()), C.c_void_p(tk.data_ptr()))


def test_noalloc_matches_allocating_entry_point_on_two_calls():
    import torch

    assert torch.cuda.is_available(), "needs a CUDA device"
    L = mlt.lib()
    stream = torch.cuda.current_stream()
    for seed, n in [(3, 40000), (4, 40000 - 123)]:
        w = W.make_workload(2, seed=seed, n=n)
        mlt.load_workload_models(w)
        x = torch.from_numpy(w.feats).cuda()
        ref_pv, ref_pf, ref_tk = mlt.screen(x, w.thr, w.k)
        mlt.sync_status()
        ref = (ref_pv.cpu().numpy(), ref_pf.cpu().numpy(), ref_tk.cpu().numpy())
        for _ in range(2):
            pv = torch.full((n,), float("nan"), device="cuda")
            pf = torch.full((n,), float("nan"), device="cuda")
            tk = torch.full((w.k,), -7, dtype=torch.int64, device="cuda")
            rc = _call(L, stream, x, n, w.thr, w.k, pv, pf, tk)
            assert rc == 0, L.mlt_last_error()
            torch.cuda.synchronize()
            assert_same_bits(pf.cpu().numpy(), ref[1], "perf (no-alloc)")
            assert_pvalid(pv.cpu().numpy(), ref[0])
            assert np.array_equal(tk.cpu().numpy(), ref[2])


def _compare_with_allocating(L, w, calls=2):
    import torch

    stream = torch.cuda.current_stream()
    mlt.load_workload_models(w)
    x = torch.from_numpy(w.feats).cuda()
    ref_pv, ref_pf, ref_tk = mlt.screen(x, w.thr, w.k)
    mlt.sync_status()
    ref = (ref_pv.cpu().numpy(), ref_pf.cpu().numpy(), ref_tk.cpu().numpy())
    for _ in range(calls):
        pv = torch.full((w.n,), float("nan"), device="cuda")
        pf = torch.full((w.n,), float("nan"), device="cuda")
        tk = torch.full((w.k,), -7, dtype=torch.int64, device="cuda")
        rc = _call(L, stream, x, w.n, w.thr, w.k, pv, pf, tk)
        assert rc == 0, L.mlt_last_error()
        mlt.sync_status()
        assert_same_bits(pf.cpu().numpy(), ref[1], "perf (no-alloc)")
        assert_pvalid(pv.cpu().numpy(), ref[0])
        assert np.array_equal(tk.cpu().numpy(), ref[2])


@pytest.mark.parametrize("n", [262144, 1, 31])
def test_noalloc_at_the_size_limit_and_on_tiny_batches(n):
    """The largest batch the static scratch holds (its ballot, tile-count
    and key arrays are full) and batches of one and 31 candidates (the
    smallest tiles the launch planner picks)."""
    _compare_with_allocating(mlt.lib(), W.make_workload(1, seed=2, n=n))


def test_noalloc_timeout_is_reported_and_the_next_call_is_exact():
    """A V-pass CTA of a no-alloc call gives up waiting (the in-path
    self-test): mlt_sync_status reports it from the static array's error
    word, and the next no-alloc call equals the allocating entry point."""
    import torch

    L = mlt.lib()
    w = W.make_workload(2, seed=6, n=30000)
    mlt.load_workload_models(w)
    x = torch.from_numpy(w.feats).cuda()
    pv = torch.empty(w.n, device="cuda")
    pf = torch.empty(w.n, device="cuda")
    tk = torch.empty(w.k, dtype=torch.int64, device="cuda")
    mlt.sync_status()
    mlt.selftest_walk_timeout(2, 20_000_000)
    assert _call(L, torch.cuda.current_stream(), x, w.n, w.thr, w.k, pv, pf, tk) == 0
    with pytest.raises(mlt.MltError) as e:
        mlt.sync_status()
    assert e.value.code == -5
    mlt.sync_status()  # reading the error cleared it
    _compare_with_allocating(L, w, calls=1)


def test_noalloc_ignores_a_poisoned_static_state():
    mlt.selftest_poison_state(5, static_scratch=True)
    _compare_with_allocating(mlt.lib(), W.make_workload(2, seed=8, n=12000), calls=1)


def test_noalloc_rejects_batches_beyond_its_static_scratch():
    import torch

    L = mlt.lib()
    w = W.make_workload(1, seed=1, n=64)
    mlt.load_workload_models(w)
    x = torch.from_numpy(w.feats).cuda()
    pv = torch.empty(64, device="cuda")
    tk = torch.empty(w.k, dtype=torch.int64, device="cuda")
    rc = _call(L, torch.cuda.current_stream(), x, 262145, w.thr, w.k, pv, pv, tk)
    assert rc == -1
    assert b"static scratch" in L.mlt_last_error()
