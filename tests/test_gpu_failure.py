"""Failure detection on the GPU without a fault: a device wait that nothing
completes runs out after its limit, the host reads the timeout, and the
device stays usable for the next screening call."""
import pytest

from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import assert_parity, gpu_screen, oracle_screen

pytestmark = pytest.mark.gpu


def test_bounded_wait_timeout_is_reported_and_the_device_stays_usable():
    import torch

    torch.cuda.synchronize()
    mlt.sync_status()  # start from a clean error word
    mlt.selftest_wait_timeout(50_000_000)  # 50 ms
    with pytest.raises(mlt.MltError) as e:
        mlt.sync_status()
    assert e.value.code == -5  # MLT_ETIMEOUT
    mlt.sync_status()  # reading the error cleared it
    w = W.make_workload(1, seed=2, n=2500)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("cid,n,cta", [(2, 20000, 0), (2, 20000, 10 ** 6), (3, 9001, 5), (1, 4096, 3)])
def test_walk_timeout_inside_a_screening_call_leaves_the_next_call_exact(cid, n, cta):
    """One V-pass CTA gives up waiting for its first tree chunk (a barrier
    phase nothing completes).  It still takes its ticket, so the scan of the
    tile counts and the selection state stay consistent: the call reports
    MLT_ETIMEOUT, its other tiles keep their results, and the next call
    matches the oracle bit for bit."""
    import torch

    w = W.make_workload(cid, seed=3, n=n)
    mlt.load_workload_models(w)
    x = torch.from_numpy(w.feats).cuda()
    mlt.sync_status()
    mlt.selftest_walk_timeout(cta, 20_000_000)  # 20 ms
    pv, pf, tk = mlt.screen(x, w.thr, w.k)
    with pytest.raises(mlt.MltError) as e:
        mlt.sync_status()
    assert e.value.code == -5
    # the stalled tile has no valid candidate; every other candidate is exact
    opv, opf, otk, os_ = oracle_screen(w)
    g = pf.cpu().numpy()
    bad = (g.view("u4") != opf.view("u4")).nonzero()[0]
    assert bad.size > 0 and bad.max() - bad.min() < 256, "only the stalled tile may differ"
    assert_parity(gpu_screen(w), (opv, opf, otk, os_))


@pytest.mark.parametrize("value", [1, 7, 0xFFFFFFFF])
def test_poisoned_selection_state_does_not_reach_the_next_call(value):
    """Tickets and counts left behind by a call that stopped part-way are
    cleared before the next call's kernels run."""
    w = W.make_workload(2, seed=5, n=15000)
    o = oracle_screen(w)
    mlt.load_workload_models(w)
    mlt.selftest_poison_state(value)
    assert_parity(gpu_screen(w), o)
