"""The compiled feature program (mlt_tune_decode_jit): decoded batches whose
rows are built by the program compiled at run time with NVRTC and then
screened as stored rows must give exactly what the interpreted in-walk
decoder gives, and what the oracle gives: random knob spaces and programs
with every opcode and special values (the decoder fuzz cases), the conv2d
space at an offset, and the explorer step, whose proposals are decoded from
an index list."""
import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_parity, gpu_screen, oracle_screen
from test_gpu_fuzz_decode import _decoder

pytestmark = pytest.mark.gpu

DEFAULT_MIN_N = 1 << 20


def _bits(a):
    a = np.asarray(a)
    return a.view(np.uint32) if a.dtype == np.float32 else a


def _same(x, y):
    for u, v in zip(x[:3], y[:3]):
        assert np.array_equal(_bits(u), _bits(v))
    assert x[3] == y[3]


def _compiled_then_interpreted(w):
    try:
        mlt.tune_decode_jit(1)
        calls = mlt.decode_jit_calls()
        compiled = gpu_screen(w)
        assert mlt.decode_jit_calls() == calls + 1, "the compiled program did not run"
        mlt.tune_decode_jit(0)
        interpreted = gpu_screen(w)
        assert mlt.decode_jit_calls() == calls + 1
    finally:
        mlt.tune_decode_jit(DEFAULT_MIN_N)
    return compiled, interpreted


def test_compiled_program_is_available():
    assert mlt.decode_jit_available()


@pytest.mark.parametrize("case", range(12))
def test_random_programs_compiled_match(case):
    d, rng = _decoder(case)
    space = d.space
    n = int(min(space, rng.integers(1, 20001)))
    first = int(rng.integers(0, space - n + 1))
    F = d.program.size
    _, sample = O.features(d.radices, d.option_values, d.program, first, min(n, 2048), threads=THREADS)
    sample = np.where(np.isfinite(sample), sample, np.nan).astype(np.float32)
    th = W._QuantileThresholds(sample)
    cfg = W.ScreenConfig(970 + case, f"jit-fuzz-{case}", n, F, 1, 1, 1, 1, 0.5, 64, None, decoded=True)
    v = W.make_ensemble(cfg, "V", th, 71 + case, n_trees=int(rng.integers(1, 30)), depth=int(rng.integers(1, 9)),
                        shape="full")
    p = W.make_ensemble(cfg, "P", th, 81 + case, n_trees=int(rng.integers(1, 30)), depth=int(rng.integers(2, 12)),
                        split_prob=0.8, shape="unbalanced")
    w = W.Workload(cfg, n, None, d, first, v, p, 0.5, 64)
    compiled, interpreted = _compiled_then_interpreted(w)
    _same(compiled, interpreted)
    assert_parity(compiled, oracle_screen(w))


def test_conv2d_space_at_an_offset():
    w = W.make_workload(4, seed=5, n=70001)
    w = W.Workload(w.cfg, w.n, None, w.decoder, 123457, w.v, w.p, w.thr, w.k)
    compiled, interpreted = _compiled_then_interpreted(w)
    _same(compiled, interpreted)
    assert_parity(compiled, oracle_screen(w))


def test_explorer_step_decodes_its_index_list_the_same_way():
    import torch

    w = W.make_workload(4, seed=6, n=1024)
    d = w.decoder
    mlt.load_workload_models(w)
    rng = np.random.default_rng(66)
    m = 5000
    parent = torch.as_tensor(rng.integers(0, d.space, size=m, dtype=np.int64)).cuda()
    ps = torch.full((m,), -np.inf, dtype=torch.float32).cuda()
    kd = torch.as_tensor(rng.integers(0, 2 ** 31, size=m, dtype=np.int64).astype(np.int32)).cuda()
    dd = torch.as_tensor(rng.integers(0, 2 ** 31, size=m, dtype=np.int64).astype(np.int32)).cuda()
    lu = torch.as_tensor(np.log(rng.random(m)).astype(np.float32)).cuda()
    out = []
    try:
        for min_n in (1, 0):
            mlt.tune_decode_jit(min_n)
            calls = mlt.decode_jit_calls()
            nxt, nsc, acc = mlt.sa_step(d.radices, d.option_values, d.program, parent, ps, kd, dd, lu, 1.0, w.thr)
            mlt.sync_status()
            assert mlt.decode_jit_calls() == calls + (1 if min_n else 0)
            out.append((nxt.cpu().numpy(), nsc.cpu().numpy(), acc.cpu().numpy()))
    finally:
        mlt.tune_decode_jit(DEFAULT_MIN_N)
    for a, b in zip(*out):
        assert np.array_equal(_bits(a), _bits(b))
