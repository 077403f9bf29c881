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
