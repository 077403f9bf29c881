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
