"""The C ABI used from plain C (tests/c_client/screen_client.c), compiled
with gcc against include/mlt.h and libmlt.so: host-only calls on any
machine, a whole screening pass on the GPU (checked against the oracle)."""
import os
import subprocess

import numpy as np
import pytest

import oracle as O
from paper_2411_10764_gb300 import _build, mlt
from paper_2411_10764_gb300 import workloads as W
from screening import THREADS, assert_parity

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def client(tmp_path_factory):
    mlt.lib()  # builds libmlt.so if needed
    lib_dir = os.path.dirname(_build.LIB_PATH)
    exe = str(tmp_path_factory.mktemp("c_client") / "screen_client")
    subprocess.run(["gcc", "-O2", "-std=c99", "-Wall", "-Werror", "-I", os.path.join(_build.ROOT, "include"),
                    os.path.join(HERE, "c_client", "screen_client.c"), "-o", exe, "-L", lib_dir, "-lmlt",
                    f"-Wl,-rpath,{lib_dir}"], check=True)
    return exe


def test_c_client_host_only_calls(client):
    r = subprocess.run([client, "check"], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    assert "check ok" in r.stdout


@pytest.mark.gpu
def test_c_client_screens_like_the_oracle(client, tmp_path):
    w = W.make_workload(2, seed=12, n=9001)
    F, n, k = w.feats.shape[1], w.n, w.k
    with open(tmp_path / "in.bin", "wb") as f:
        f.write(np.int32(F).tobytes() + np.int64(n).tobytes() + np.float32(w.thr).tobytes() + np.int32(k).tobytes())
        for e in (w.v, w.p):
            f.write(np.int32(e.n_trees).tobytes() + np.int32(e.depth).tobytes())
            f.write(np.ascontiguousarray(e.nodes).tobytes())
        f.write(np.ascontiguousarray(w.feats, np.float32).tobytes())
    r = subprocess.run([client, str(tmp_path / "in.bin"), str(tmp_path / "out.bin")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    out = np.fromfile(tmp_path / "out.bin", dtype=np.uint8)
    pv = out[: 4 * n].view(np.float32)
    pf = out[4 * n: 8 * n].view(np.float32)
    tk = out[8 * n:].view(np.int64)
    opv, opf, valid, _ = O.screen_rows(w.feats, w.v, w.p, w.thr, threads=THREADS)
    otk, s = O.topk(opf, valid, k)
    assert_parity((pv, pf, tk, s), (opv, opf, otk, s))
