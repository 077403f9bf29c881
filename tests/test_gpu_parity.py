"""GPU parity: the CUDA library against the oracle, element by element, on the
same seeded inputs.  Decisions, survivor sets, top-k lists and P scores are
bit-exact (fp32 leaf sums in tree order on both sides); pvalid is within
1e-6 relative (device expf vs. host exp)."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import (THREADS, assert_parity, assert_pvalid, assert_same_bits, gpu_screen, near_counts,
                       oracle_screen, oracle_screen_chunked)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    import torch

    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    mlt.lib()


# sizes that span several 256-candidate tiles and end on a ragged tile
SMALL = {1: 4096, 2: 20000, 3: 9001, 4: 30000, 5: 5003}


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_small_workloads_match_oracle(cid):
    w = W.make_workload(cid, seed=1, n=SMALL[cid])
    if w.decoder is not None:
        w.first_index = 1234567
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("cid", [1, 3])
def test_second_seed(cid):
    w = W.make_workload(cid, seed=7, n=3000)
    assert_parity(gpu_screen(w), oracle_screen(w))


def test_empty_batch():
    w = W.make_workload(1, seed=1, n=0)
    pv, pf, tk, s = gpu_screen(w)
    assert pv.size == 0 and pf.size == 0 and s == 0
    assert np.all(tk == -1)


@pytest.mark.parametrize("n", [1, 31, 32, 33, 255, 257])
def test_tiny_and_ragged_batches(n):
    w = W.make_workload(1, seed=3, n=n)
    assert_parity(gpu_screen(w, k=8), oracle_screen(w, k=8))


@pytest.mark.parametrize("k", [1, 7, 2048, 16384])
def test_k_sizes_including_more_than_survivors(k):
    w = W.make_workload(2, seed=1, n=5000)
    assert_parity(gpu_screen(w, k=k), oracle_screen(w, k=k))


@pytest.fixture(scope="module")
def mid():
    w = W.make_workload(2, seed=4, n=20000)
    return w, oracle_screen(w, k=8000)


@pytest.mark.parametrize("k", [2, 63, 300, 511, 512, 513, 1000, 4099])
def test_k_sizes_around_the_ordering_switch(mid, k):
    """Up to 512 selected keys are ordered by counting, more by a sort."""
    w, (opv, opf, otk, os_) = mid
    assert_parity(gpu_screen(w, k=k), (opv, opf, otk[:k], os_))


@pytest.fixture(scope="module")
def all_tied():
    """30,000 copies of one surviving candidate: every key shares its score,
    so the whole collection (more than shared memory holds) sits in the
    boundary bucket and the selection runs down to the position digits."""
    w = W.make_workload(2, seed=1, n=2000)
    _, _, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    row = w.feats[int(np.nonzero(valid)[0][0])]
    x = np.ascontiguousarray(np.tile(row, (30000, 1)))
    return w, x, oracle_screen(w, feats=x, k=16384)


@pytest.mark.parametrize("k", [1, 100, 512, 513, 4096, 16384])
def test_topk_when_every_score_ties(all_tied, k):
    w, x, (opv, opf, otk, os_) = all_tied
    assert os_ == 30000
    assert np.array_equal(otk[:k], np.arange(k))
    assert_parity(gpu_screen(w, feats=x, k=k), (opv, opf, otk[:k], os_))


@pytest.mark.parametrize("thr", [1e-6, 0.999999, 0.3, 0.75])
def test_thresholds_all_none_some(thr):
    w = W.make_workload(1, seed=1, n=4096)
    assert_parity(gpu_screen(w, thr=thr), oracle_screen(w, thr=thr))


def test_missing_values_in_full_tables():
    w = W.make_workload(1, seed=1, n=6000)
    rng = np.random.default_rng(5)
    x = w.feats.copy()
    x[rng.random(size=x.shape) < 0.25] = np.nan
    x[rng.random(size=x.shape) < 0.02] = np.inf
    x[rng.random(size=x.shape) < 0.02] = -np.inf
    x[:3] = np.nan  # rows entirely missing
    assert_parity(gpu_screen(w, feats=x), oracle_screen(w, feats=x))


def test_duplicate_rows_tie_break_by_index():
    w = W.make_workload(2, seed=1, n=8000)
    x = w.feats.copy()
    x[1::2] = x[0::2]  # every score appears twice
    x[5000:] = x[17]  # a large block of identical candidates
    g = gpu_screen(w, feats=x, k=512)
    o = oracle_screen(w, feats=x, k=512)
    assert_parity(g, o)


def test_unbalanced_shallow_trees_use_padded_full_tables():
    cfg = W.ScreenConfig(98, "unbalanced-d7", 7000, 40, 60, 7, 90, 7, 0.5, 100, None,
                         shape="unbalanced", split_dist="zipf", nan_frac=0.2, dup_frac=0.05)
    x = W.make_features(W.CONFIGS[5], 2, 7000)[:, :40].copy()
    th = W._QuantileThresholds(x[:4096])
    w = W.Workload(cfg, 7000, x, None, 0, W.make_ensemble(cfg, "V", th, 4),
                   W.make_ensemble(cfg, "P", th, 4), 0.5, 100)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("F", [30, 7])
def test_feature_counts_not_multiple_of_four(F):
    cfg = W.ScreenConfig(97, f"f{F}", 3000, F, 40, 6, 50, 5, 0.5, 64, None)
    x = W.make_features(W.CONFIGS[1], 3, 3000)
    x = np.ascontiguousarray(np.tile(x, (1, 2))[:, :F])
    th = W._QuantileThresholds(x[:2048])
    w = W.Workload(cfg, 3000, x, None, 0, W.make_ensemble(cfg, "V", th, 5),
                   W.make_ensemble(cfg, "P", th, 5), 0.5, 64)
    assert_parity(gpu_screen(w), oracle_screen(w))


def test_unaligned_feature_pointer():
    import torch

    w = W.make_workload(1, seed=1, n=2000)
    mlt.load_workload_models(w)
    buf = torch.empty(w.feats.size + 1, dtype=torch.float32, device="cuda")
    x = buf[1:].view(w.feats.shape)  # 4-byte aligned only
    x.copy_(torch.from_numpy(w.feats))
    pv, pf, tk = mlt.screen(x, w.thr, w.k)
    mlt.sync_status()
    g = (pv.cpu().numpy(), pf.cpu().numpy(), tk.cpu().numpy(), mlt.last_survivor_count())
    assert_parity(g, oracle_screen(w))


def test_host_buffer_entry_point_matches_device_call():
    w = W.make_workload(2, seed=2, n=12345)
    g = gpu_screen(w)
    pv, pf, tk = mlt.screen_host(w.feats, w.thr, w.k)
    assert_same_bits(pv, g[0], "pvalid (host entry)")
    assert_same_bits(pf, g[1], "perf (host entry)")
    assert np.array_equal(tk, g[2])


def test_decoded_knobs_and_features_bit_exact():
    d = W.conv2d_decoder(seed=1)
    for first, n in [(0, 4096), (16777216 - 5000, 5000), (987654, 3333)]:
        knobs, feats = mlt.decode_knobs(d.radices, d.option_values, d.program, first, n)
        ok, of = O.features(d.radices, d.option_values, d.program, first, n, threads=THREADS)
        assert np.array_equal(knobs.cpu().numpy(), ok)
        assert_same_bits(feats.cpu().numpy(), of, "decoded features")


def test_decoded_screen_equals_materialised_screen():
    w = W.make_workload(4, seed=1, n=20000)
    w.first_index = 5_000_000
    d = w.decoder
    g_dec = gpu_screen(w)
    _, feats = mlt.decode_knobs(d.radices, d.option_values, d.program, w.first_index, w.n)
    import torch

    pv, pf, tk = mlt.screen(feats, w.thr, w.k)
    assert_same_bits(pf.cpu().numpy(), g_dec[1], "perf decoded vs materialised")
    assert np.array_equal(tk.cpu().numpy() + w.first_index, g_dec[2])
    torch.cuda.synchronize()


def test_full_size_workload2_all_outputs():
    w = W.make_workload(2, seed=1)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("cid", [3, 4, 5])
def test_full_size_all_outputs(cid):
    """Workloads 3, 4 (all 16,777,216 decoded indices) and 5 at full size,
    in the launch configuration the benchmark times, against the oracle run
    over the whole pool on every host core: survivor count, every P score
    and V decision bit for bit, every pvalid within 1e-6, and the top-k list
    against the oracle's own full sort."""
    w = W.make_workload(cid, seed=1)
    gpu = gpu_screen(w)
    opv, opf, otk, os_, omv = oracle_screen_chunked(w)
    assert_parity(gpu, (opv, opf, otk, os_))
    near_tau, near_k = near_counts(omv, O.tau(w.thr), opf, otk, w.first_index)
    print(f"workload {cid}: {w.n} candidates, {os_} valid; {near_tau} V margins within 1e-6 of the cut, "
          f"{near_k} P scores within 1e-6 of the k-th kept score")


# --------------------------------------------------------------------------
# Model A rerank of the kept candidates
# --------------------------------------------------------------------------

def _gpu_rerank(w, a, cand, n_final):
    import torch

    mlt.load_ensemble(mlt.MLT_MODEL_A, a.nodes, a.n_trees, a.depth)
    x = torch.from_numpy(w.feats).cuda()
    c = torch.as_tensor(np.asarray(cand, np.int64)).cuda()
    sc, fin = mlt.rerank(x, c, n_final)
    mlt.sync_status()
    return sc.cpu().numpy(), fin.cpu().numpy()


@pytest.mark.parametrize("cid,shape,depth", [(2, "unbalanced", 14), (3, "unbalanced", 12), (1, "full", 8)])
def test_rerank_of_screened_topk_matches_oracle(cid, shape, depth):
    import torch

    w = W.make_workload(cid, seed=2, n=12000)
    a = W.make_ensemble(w.cfg, "A", W._QuantileThresholds(w.feats[:4096]), 3, n_trees=150, depth=depth,
                        split_prob=0.8, shape=shape)
    mlt.load_workload_models(w)
    _, _, tk = mlt.screen(torch.from_numpy(w.feats).cuda(), w.thr, w.k)
    cand = tk.cpu().numpy()
    n_final = w.k // 2  # (alpha + 1) N kept, N final, alpha = 1
    sc, fin = _gpu_rerank(w, a, cand, n_final)
    osc, ofin = O.rerank(w.feats, cand, a, n_final)
    assert_same_bits(sc, osc, "A scores")
    assert np.array_equal(fin, ofin)


def test_rerank_edge_cases():
    w = W.make_workload(1, seed=4, n=3000)
    a = W.make_model_a(w, n_trees=40, depth=10)
    mlt.load_workload_models(w)
    cases = [
        ([17], 1),
        ([5, -1, 5, 2999, 0, -1], 8),  # padding, a duplicate, n_final past the valid entries
        ([-1, -1], 3),
        (list(range(0, 3000, 7)), 64),
    ]
    for cand, n_final in cases:
        sc, fin = _gpu_rerank(w, a, cand, n_final)
        osc, ofin = O.rerank(w.feats, np.asarray(cand, np.int64), a, n_final)
        assert_same_bits(sc, osc, "A scores")
        assert np.array_equal(fin, ofin)


def test_rerank_reports_out_of_range_index():
    import torch

    w = W.make_workload(1, seed=4, n=100)
    a = W.make_model_a(w, n_trees=10, depth=6)
    mlt.load_workload_models(w)
    mlt.load_ensemble(mlt.MLT_MODEL_A, a.nodes, a.n_trees, a.depth)
    x = torch.from_numpy(w.feats).cuda()
    c = torch.tensor([3, 100, 7], dtype=torch.int64, device="cuda")
    sc, fin = mlt.rerank(x, c, 3)
    with pytest.raises(mlt.MltError) as e:
        mlt.sync_status()
    assert e.value.code == -1
    assert np.isneginf(sc.cpu().numpy()[1])
    mlt.sync_status()  # the error was cleared


# --------------------------------------------------------------------------
# Batched accumulation: screen batch after batch until enough survivors
# --------------------------------------------------------------------------

def _expected_prefix(valid, n, batch, target):
    """(consumed, kept, batches) of the accumulation rule on oracle decisions."""
    kept = 0
    for b, b0 in enumerate(range(0, n, batch)):
        b1 = min(n, b0 + batch)
        kept += int(valid[b0:b1].sum())
        if kept >= target:
            return b1, kept, b + 1
    return n, kept, -(-n // batch)


@pytest.mark.parametrize("target,batch", [(1, 4096), (3000, 4096), (9000, 3000), (10 ** 9, 4096), (5000, 20000)])
def test_screen_until_equals_oracle_on_the_consumed_prefix(target, batch):
    import torch

    w = W.make_workload(2, seed=3, n=20000)
    mlt.load_workload_models(w)
    pv, pf, tk, stats = mlt.screen_until(torch.from_numpy(w.feats).cuda(), batch, target, w.thr, w.k)
    mlt.sync_status()
    opv, opf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    consumed, kept, batches = _expected_prefix(valid, w.n, batch, target)
    assert stats.cpu().tolist() == [consumed, kept, batches]
    want, _ = O.topk(opf[:consumed], valid[:consumed], w.k)
    assert np.array_equal(tk.cpu().numpy(), want)
    assert_same_bits(pf.cpu().numpy()[:consumed], opf[:consumed], "perf (consumed prefix)")
    assert_pvalid(pv.cpu().numpy()[:consumed], opv[:consumed])


def test_screen_until_decoded_space():
    w = W.make_workload(4, seed=1, n=30000)
    d = w.decoder
    first, batch, target = 777777, 8192, 6000
    mlt.load_workload_models(w)
    pv, pf, tk, stats = mlt.screen_until_decoded(d.radices, d.option_values, d.program, first, w.n, batch,
                                                 target, w.thr, w.k)
    mlt.sync_status()
    _, x = O.features(d.radices, d.option_values, d.program, first, w.n, threads=THREADS)
    opv, opf, valid, _ = O.screen_rows(x, w.v, w.p, w.thr, threads=THREADS)
    consumed, kept, batches = _expected_prefix(valid, w.n, batch, target)
    assert stats.cpu().tolist() == [consumed, kept, batches]
    want, _ = O.topk(opf[:consumed], valid[:consumed], w.k, index_base=first)
    assert np.array_equal(tk.cpu().numpy(), want)
    assert_same_bits(pf.cpu().numpy()[:consumed], opf[:consumed], "perf (consumed prefix)")


def test_screen_until_without_per_candidate_outputs_and_repeat():
    import torch

    w = W.make_workload(1, seed=6, n=10000)
    mlt.load_workload_models(w)
    x = torch.from_numpy(w.feats).cuda()
    first = mlt.screen_until(x, 1000, 2500, w.thr, w.k, with_outputs=False)
    second = mlt.screen_until(x, 1000, 2500, w.thr, w.k, with_outputs=False)
    mlt.sync_status()
    assert np.array_equal(first[2].cpu().numpy(), second[2].cpu().numpy())
    assert first[3].cpu().tolist() == second[3].cpu().tolist()
    _, opf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr)
    consumed, kept, batches = _expected_prefix(valid, w.n, 1000, 2500)
    assert first[3].cpu().tolist() == [consumed, kept, batches]
    want, _ = O.topk(opf[:consumed], valid[:consumed], w.k)
    assert np.array_equal(first[2].cpu().numpy(), want)


# --------------------------------------------------------------------------
# Explorer proposal step (one simulated-annealing move per chain)
# --------------------------------------------------------------------------

def _gpu_sa(radices, options, program, parent, ps, kd, dd, lu, temperature, thr):
    import torch

    t = lambda a, dt: torch.as_tensor(np.ascontiguousarray(a).astype(dt)).cuda()
    nxt, nsc, acc = mlt.sa_step(radices, options, program, t(parent, np.int64), t(ps, np.float32),
                                t(np.asarray(kd, np.uint32).view(np.int32), np.int32),
                                t(np.asarray(dd, np.uint32).view(np.int32), np.int32), t(lu, np.float32),
                                temperature, thr)
    mlt.sync_status()
    return nxt.cpu().numpy(), nsc.cpu().numpy(), acc.cpu().numpy()


def test_sa_step_hand_worked_on_gpu():
    from conftest import floats, golden, slots_to_nodes

    g = golden("sa_step.json")
    prog = np.zeros(len(g["program"]), mlt.OP_DTYPE)
    for i, (op, a, b, c) in enumerate(g["program"]):
        prog[i] = (op, a, b, c)
    mlt.set_num_features(2)
    mlt.load_ensemble(mlt.MLT_MODEL_V, slots_to_nodes(g["V"], mlt.NODE_DTYPE), 1, 1)
    mlt.load_ensemble(mlt.MLT_MODEL_P, slots_to_nodes(g["P"], mlt.NODE_DTYPE), 1, 1)
    for case in g["cases"]:
        nxt, nsc, acc = _gpu_sa(g["radices"], np.array(g["options"], np.float32), prog, g["parent"],
                                floats(g["parent_score"]), g["knob_draw"], g["digit_draw"], floats(g["log_u"]),
                                case["temperature"], g["thr"])
        assert nxt.tolist() == case["next"]
        assert_same_bits(nsc, floats(case["score"]), "chain scores")
        assert acc.tolist() == case["accepted"]


def test_sa_chains_match_oracle_over_three_steps():
    w = W.make_workload(4, seed=1, n=1000)
    d = w.decoder
    mlt.load_workload_models(w)
    rng = np.random.default_rng(12)
    m = 6000
    parent = rng.integers(0, d.space, size=m).astype(np.int64)
    parent[::97] = -1  # inactive chains
    ps = np.full(m, -np.inf, np.float32)
    for step, temperature in enumerate([2.0, 1.0, 0.25]):
        kd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
        dd = rng.integers(0, 2 ** 32, size=m, dtype=np.uint64).astype(np.uint32)
        lu = np.log(rng.random(m)).astype(np.float32)
        g = _gpu_sa(d.radices, d.option_values, d.program, parent, ps, kd, dd, lu, temperature, w.thr)
        o = O.sa_step(d.radices, d.option_values, d.program, w.v, w.p, parent, ps, kd, dd, lu, temperature, w.thr)
        assert np.array_equal(g[0], o[0]), step
        assert_same_bits(g[1], o[1], f"chain scores step {step}")
        assert np.array_equal(g[2], o[2]), step
        parent, ps = o[0], o[1]
    assert 0 < int(g[2].sum()) < m


def test_sa_step_reports_parent_past_the_space():
    w = W.make_workload(4, seed=1, n=100)
    d = w.decoder
    mlt.load_workload_models(w)
    with pytest.raises(mlt.MltError) as e:
        _gpu_sa(d.radices, d.option_values, d.program, [3, d.space], [0.0, 0.0], [1, 1], [1, 1], [-1.0, -1.0],
                1.0, w.thr)
    assert e.value.code == -1
    mlt.sync_status()


def test_host_batches_pipeline_matches_oracle():
    """Pipelined host batches (mlt_screen_host_batches): every batch equals
    the oracle's screening of it, whatever the overlap; optional outputs
    may be skipped."""
    import torch

    w = W.make_workload(2, seed=9, n=20001)
    mlt.load_workload_models(w)
    rng = np.random.default_rng(5)
    batches = [np.ascontiguousarray(w.feats[rng.permutation(w.n)]) for _ in range(5)]
    pinned = [torch.from_numpy(b).pin_memory().numpy() for b in batches]
    outs = mlt.screen_host_batches(pinned, w.thr, w.k)
    for b, (pv, pf, tk) in zip(batches, outs):
        opv, opf, valid, _ = O.screen_rows(b, w.v, w.p, w.thr, threads=THREADS)
        otk, s = O.topk(opf, valid, w.k)
        assert_parity((pv, pf, tk, s), (opv, opf, otk, s))
    # top-k only, a single batch, then an odd batch count
    for nb in (1, 3):
        outs = [(None, None, np.empty(w.k, np.int64)) for _ in range(nb)]
        outs = mlt.screen_host_batches(pinned[:nb], w.thr, w.k, outs=outs)
        for b, (_, _, tk) in zip(batches, outs):
            _, opf, valid, _ = O.screen_rows(b, w.v, w.p, w.thr, threads=THREADS)
            otk, _ = O.topk(opf, valid, w.k)
            assert np.array_equal(tk, otk)


@pytest.mark.parametrize("F,depth,shape", [(1, 6, "full"), (1024, 8, "full"), (1024, 12, "unbalanced"),
                                           (1, 11, "unbalanced"), (1000, 10, "full")])
def test_feature_count_extremes(F, depth, shape):
    """The smallest and largest feature rows (1 and 1,024 fp32 features),
    with full tables and with the deep-tree (compact) walk."""
    rng = np.random.default_rng(F + depth)
    n = 2500
    x = rng.lognormal(0.0, 1.0, size=(n, F)).astype(np.float32)
    x[rng.random((n, F)) < 0.05] = np.nan
    cfg = W.ScreenConfig(98, f"f{F}", n, F, 30, depth, 40, depth, 0.5, 100, None, shape=shape)
    th = W._QuantileThresholds(x[:2048])
    w = W.Workload(cfg, n, x, None, 0, W.make_ensemble(cfg, "V", th, 7, split_prob=0.8),
                   W.make_ensemble(cfg, "P", th, 8, split_prob=0.8), 0.5, 100)
    assert_parity(gpu_screen(w), oracle_screen(w))


@pytest.mark.parametrize("v_trees,p_trees,depth,shape", [(1, 1, 1, "full"), (1, 3, 14, "unbalanced"),
                                                         (5000, 3000, 3, "full"), (700, 900, 14, "unbalanced")])
def test_tree_count_and_depth_extremes(v_trees, p_trees, depth, shape):
    """Stumps and single trees, thousands of shallow trees (many chunks), and
    the deepest ensembles the library takes (depth 14, compact tables)."""
    rng = np.random.default_rng(v_trees + depth)
    n, F = 3001, 24
    x = rng.lognormal(0.0, 1.0, size=(n, F)).astype(np.float32)
    cfg = W.ScreenConfig(99, "trees", n, F, v_trees, depth, p_trees, depth, 0.5, n, None, shape=shape)
    th = W._QuantileThresholds(x[:2048])
    w = W.Workload(cfg, n, x, None, 0, W.make_ensemble(cfg, "V", th, 3, split_prob=0.8),
                   W.make_ensemble(cfg, "P", th, 4, split_prob=0.8), 0.5, n)  # k = n: the whole order
    assert_parity(gpu_screen(w), oracle_screen(w))
