"""GPU parity of the walk-rate ceiling kernel (mlt_walk_peak): the sums it
leaves are the oracle's sequential fp32 sums over the resident trees
repeated `rounds` times, bit for bit, so the timed walk is the screening
walk doing real work."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_same_bits

pytestmark = pytest.mark.gpu


def _expected(ens, x, resident, rounds):
    nodes = ens.nodes.reshape(ens.n_trees, -1)[:resident]
    rep = W.Ensemble(np.ascontiguousarray(np.tile(nodes, (rounds, 1)).reshape(-1)), resident * rounds, ens.depth)
    return O.margins(rep, x, threads=THREADS)


@pytest.mark.parametrize("cid,n,rounds,model", [(2, 5001, 3, "V"), (2, 777, 2, "P"), (3, 2049, 1, "V"),
                                                (1, 3000, 2, "P")])
def test_walk_peak_sums_match_oracle(cid, n, rounds, model):
    import torch

    w = W.make_workload(cid, seed=2, n=n)
    x = w.feats.copy()
    if cid == 1:
        x[::7, ::3] = np.nan  # missing values take each node's default side
    mlt.load_workload_models(w)
    ens = w.v if model == "V" else w.p
    mid = mlt.MLT_MODEL_V if model == "V" else mlt.MLT_MODEL_P
    sums, visits = mlt.walk_peak(torch.from_numpy(x).cuda(), rounds, model_id=mid)
    mlt.sync_status()
    resident = visits // (n * ens.depth * rounds)
    assert visits == n * resident * ens.depth * rounds
    assert 1 <= resident <= ens.n_trees
    assert_same_bits(sums.cpu().numpy(), _expected(ens, x, resident, rounds), "walk-peak sums")


def test_walk_peak_rejects_compact_tables():
    import torch

    w = W.make_workload(5, seed=1, n=100)
    mlt.load_workload_models(w)
    with pytest.raises(mlt.MltError) as e:
        mlt.walk_peak(torch.from_numpy(w.feats).cuda(), 1)
    assert e.value.code == -1
