"""Benchmark: candidates screened per second (V filter + P score + top-k) on
GB300, with roofline, CPU-oracle baseline and end-to-end figures.

One step = one screening call over one batch of a workload (ML^2Tuner's
explorer step, Sec. 2; tree ensembles as in Table 3).  The headline line is
the largest single-GPU workload, the exhaustive conv2d knob space: all
16,777,216 candidate indices of 8 knobs x 8 options are decoded on the
device into 96 fp32 features inside the walk kernels, V = 300 trees of depth
10, P = 600 trees of depth 10, validity threshold 0.5, top-1,024.  The same
line carries a `per_config` record for every workload (1 tiny, 2 gemm,
3 sa-batch, 4 conv2d decoded, 5 skewed-nan).  Inputs sit in HBM before the
timed region; L2 is flushed (a 256 MB device write) before every timed
step, outside its events.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload 1-5] [--no-per-config]

Under torchrun every rank screens its own batch (different seed): weak
scaling, no collective on the data path; rank 0 prints the JSON line with
the max-over-ranks time (the per-workload records and the next-row timings
are taken at N = 1 only).  `--impl reference` times the CPU oracle instead
(rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "candidates screened/sec (V filter + P score + top-k) at 1 GB300; % HBM roofline"
DEFAULT_WORKLOAD = 4  # the largest single-GPU configuration
ALL_WORKLOADS = (1, 2, 3, 4, 5)
L2_FLUSH_BYTES = 256 << 20
SM_COUNT = 152
SM_MAX_MHZ_NOMINAL = 2070.0
MIN_TIMED_S = 0.4  # per-workload records: enough steps for clock samples


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p.get("sm_max_mhz", SM_MAX_MHZ_NOMINAL)), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, SM_MAX_MHZ_NOMINAL, "fallback"


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    QUERY = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()
        time.sleep(0.3)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        rows = [l.split(", ") for l in self.lines if l.count(",") >= 9]
        mine = [r for r in rows if self.uuid and r[1].strip() == self.uuid] or rows
        sm = [float(r[2]) for r in mine if r[2].replace(".", "").isdigit()]
        mx = [float(r[3]) for r in mine if r[3].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in mine for i in range(4) if r[6 + i].strip() == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons, "samples": len(mine)}


# ---------------------------------------------------------------------------
# the oracle on the host cores
# ---------------------------------------------------------------------------
def oracle_pass(w, rows: int):
    """One whole oracle pass over the workload's first `rows` candidates:
    (decode +) V screen + P score + top-k, single thread."""
    import oracle as O

    if w.decoder is None:
        x = w.feats[:rows]
    else:
        d = w.decoder
        _, x = O.features(d.radices, d.option_values, d.program, w.first_index, rows)
    return O.screen(x, w.v, w.p, w.thr, w.k)


def oracle_rate(w, budget_s: float):
    """Single-threaded oracle throughput (candidates/s) on leading rows of
    the workload: whole oracle passes (screen + top-k) until `budget_s`
    seconds have been spent (the whole workload if one pass fits a quarter
    of the budget, else a leading slice)."""
    probe = min(w.n, 1024)
    t0 = time.perf_counter()
    oracle_pass(w, probe)
    per_row = (time.perf_counter() - t0) / probe
    n = min(w.n, int(max(probe, budget_s / 4 / max(per_row, 1e-9))))
    done, calls, t0 = 0, 0, time.perf_counter()
    while True:
        oracle_pass(w, n)
        done += n
        calls += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return done / el, {"rows_per_call": n, "calls": calls, "seconds": round(el, 3)}


def cpu_baseline(w, budget_s: float):
    rate, info = oracle_rate(w, budget_s)
    what = "decode, V, P, sort" if w.decoder is not None else "V, P, sort"
    return {"value": rate, "unit": "candidates/s", "cores": 1, "host_cores": host_cores(), "kind": "oracle",
            "sample": f"first {info['rows_per_call']} of {w.n} candidates x {info['calls']} whole oracle passes "
                      f"({what}), {info['seconds']} s on one of the host's {host_cores()} cores"}


def config_dict(w, seed: int, world: int):
    """The workload a line measures; both arms write the same dict."""
    c = w.cfg
    return {"workload": f"{c.name} (workload {c.id})", "n": w.n, "F": c.F,
            "v_trees": c.v_trees, "v_depth": c.v_depth, "p_trees": c.p_trees, "p_depth": c.p_depth,
            "thr": c.thr, "k": c.k, "seed": seed, "parallelism": f"replicas x{world}",
            "l2": "flushed before every timed step (256 MB device write, outside the step events)"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return 0
    from paper_2411_10764_gb300 import workloads as W

    w = W.make_workload(args.workload, seed=args.seed, n=args.n)
    import oracle as O

    O.build()
    # size one step so that warmup + steps stay near 60 s of oracle work
    probe = min(w.n, 1024)
    t0 = time.perf_counter()
    oracle_pass(w, probe)
    per_row = (time.perf_counter() - t0) / probe
    rows = int(max(64, min(w.n, 60.0 / max(1, args.steps + args.warmup) / max(per_row, 1e-9))))
    for _ in range(args.warmup):
        oracle_pass(w, rows)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle_pass(w, rows)
        times.append(time.perf_counter() - t0)
    mean = sum(times) / len(times)
    value = rows / mean
    what = "decode, V, P, sort" if w.decoder is not None else "V, P, sort"
    sample = (f"first {rows} of {w.n} candidates per step (whole oracle pass: {what}), one of the host's "
              f"{host_cores()} cores")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "candidates/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": mean * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded; shapes of the paper's tuning tasks)",
        "config": config_dict(w, args.seed, world),
        "cpu_baseline": {"value": value, "unit": "candidates/s", "cores": 1, "host_cores": host_cores(),
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": "candidates/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# roofline bookkeeping
# ---------------------------------------------------------------------------
def walk_source_hash() -> str:
    """Hash of the sources the tree-walk kernels compile from (the walk
    device code, the launch planners and instantiations, the internal
    header, which also holds the batch size from which decoded steps use the
    compiled feature program) and of that program's generator, in a fixed
    order."""
    import glob
    import hashlib

    csrc = os.path.join(ROOT, "paper_2411_10764_gb300", "csrc")
    files = [os.path.join(csrc, "walk.cuh"), os.path.join(csrc, "mlt_internal.cuh")]
    files += sorted(glob.glob(os.path.join(csrc, "traverse*.cu")))
    files += [os.path.join(csrc, "jit_decode.cu")]
    h = hashlib.sha256()
    for path in files:
        with open(path, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def dram_traffic(workload: int, phase: str):
    """DRAM bytes per launch of the phase's walk kernel from the committed
    ncu capture, or None if there is none or the walk sources changed since."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            tr = json.load(f)
    except (OSError, ValueError):
        return None
    if tr.get("walk_source_hash") != walk_source_hash():
        return None
    ent = tr.get(f"workload{workload}:{phase}")
    return ent.get("dram_bytes_per_launch") if ent else None


def mean_path(ens, x):
    """Mean number of split nodes a row of `x` passes through per tree
    (the walk's node visits), counted by walking the heap-ordered trees
    with numpy.  For full trees this is the depth."""
    t = ens.nodes.reshape(ens.n_trees, -1)
    feat, val, dl = t["feature"], t["value"], t["default_left"].astype(bool)
    tree = np.arange(ens.n_trees)[None, :]
    node = np.zeros((x.shape[0], ens.n_trees), np.int64)
    rows = np.arange(x.shape[0])[:, None]
    visits = 0
    for _ in range(ens.depth):
        f = feat[tree, node]
        active = f >= 0
        if not active.any():
            break
        xv = x[rows, np.maximum(f, 0)]
        left = np.where(np.isnan(xv), dl[tree, node], xv < val[tree, node])
        node = np.where(active, 2 * node + 1 + (~left), node)
        visits += int(active.sum())
    return visits / (x.shape[0] * ens.n_trees)


def algorithmic_counts(w, survivors, survived_rows=None):
    """Node visits and algorithmic HBM bytes of one step.  Full trees:
    trees x depth visits per candidate; unbalanced trees: trees x the mean
    path length over a 2,048-row sample (the P pass's over the sample's
    survivors).  Bytes: the feature matrix (0 when decoded on chip), 8 B per
    split node and 4 B per leaf of each table."""
    c = w.cfg
    if c.shape == "full":
        v_path, p_path = float(c.v_depth), float(c.p_depth)
    else:
        xs = w.feats[:2048]
        v_path = mean_path(w.v, xs)
        keep = xs if survived_rows is None else xs[survived_rows[:xs.shape[0]]]
        p_path = mean_path(w.p, keep if keep.shape[0] else xs)
    v_visits = w.n * c.v_trees * v_path
    p_visits = survivors * c.p_trees * p_path
    feat_bytes = 0 if w.feats is None else w.feats.nbytes

    def table(ens):
        f = ens.nodes["feature"]
        return int((f >= 0).sum()) * 8 + int((f == -1).sum()) * 4

    v_table, p_table = table(w.v), table(w.p)
    out_bytes = w.n * 8 + c.k * 8
    return {"v_visits": v_visits, "p_visits": p_visits, "v_path": v_path, "p_path": p_path,
            "feat_bytes": feat_bytes,
            "v_table_bytes": v_table, "p_table_bytes": p_table, "out_bytes": out_bytes,
            "survivor_feat_bytes": 0 if w.feats is None else survivors * c.F * 4}


def near_counts(pv, pf, tk, thr, first_index, rel=1e-6):
    """Candidates near a decision, from the device outputs: V margins within
    1e-6 of the validity cut (read through pvalid = sigmoid(margin): a
    margin step of 1e-6 moves pvalid by thr (1 - thr) 1e-6), and survivors
    whose P score lies within 1e-6 (relative) of the k-th kept score."""
    near_tau = int(np.sum(np.abs(pv.astype(np.float64) - thr) <= rel * thr * (1.0 - thr)))
    kept = tk[tk >= 0] - first_index
    near_k = 0
    if kept.size:
        kth = float(pf[kept[-1]])
        fin = pf[np.isfinite(pf)].astype(np.float64)
        near_k = int(np.sum(np.abs(fin - kth) <= rel * abs(kth)))
    return {"near_cut": near_tau, "near_kth": near_k,
            "how": "from the device outputs: |pvalid - thr| <= 1e-6 thr (1 - thr) (a V margin within 1e-6 of the "
                   "cut), |perf - perf[k-th]| <= 1e-6 |perf[k-th]|; decisions and scores are bit-exact against "
                   "the oracle in the full-size parity tests"}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
class Ctx:
    def __init__(self, dev, stream, world, rank, dist):
        import torch

        self.dev, self.stream, self.world, self.rank, self.dist = dev, stream, world, rank, dist
        self.flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
        self.uuid = None
        try:
            self.uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
        except Exception:
            pass

    def max_over_ranks(self, v: float) -> float:
        if self.dist is None:
            return v
        import torch

        t = torch.tensor([v], dtype=torch.float64, device=self.dev)
        self.dist.all_reduce(t, op=self.dist.ReduceOp.MAX)
        return float(t.item())


def screen_step(ctx, w):
    """(step function, device inputs/outputs) for one screening call."""
    import torch
    from paper_2411_10764_gb300 import mlt

    n, k, thr = w.n, w.k, w.thr
    pv = torch.empty(n, dtype=torch.float32, device=ctx.dev)
    pf = torch.empty(n, dtype=torch.float32, device=ctx.dev)
    tk = torch.empty(k, dtype=torch.int64, device=ctx.dev)
    d = w.decoder
    x = None if d is not None else torch.from_numpy(w.feats).to(ctx.dev)

    def step():
        if d is None:
            mlt.screen(x, thr, k, pv, pf, tk, stream=ctx.stream)
        else:
            # knob indices decoded and featurised inside the walk kernels
            mlt.screen_decoded(d.radices, d.option_values, d.program, w.first_index, n, thr, k,
                               out_pvalid=pv, out_perf=pf, out_topk=tk, stream=ctx.stream)

    return step, {"x": x, "pv": pv, "pf": pf, "tk": tk}


def timed_steps(ctx, step, steps, sample_clocks):
    """Time exactly `steps` calls with CUDA events on the launching stream,
    L2 flushed before each (outside the events).  Returns (ms per step over
    ranks, clocks, launches, wall s)."""
    import torch
    from paper_2411_10764_gb300 import mlt

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    sampler = ClockSampler(ctx.uuid) if sample_clocks else None
    if ctx.dist is not None:
        ctx.dist.barrier()
    torch.cuda.synchronize(ctx.dev)
    if sampler:
        sampler.start()
    launches0 = mlt.kernel_launches()
    wall0 = time.perf_counter()
    for i in range(steps):
        ctx.flush.fill_(float(i))
        starts[i].record(ctx.stream)
        step()
        ends[i].record(ctx.stream)
    torch.cuda.synchronize(ctx.dev)
    wall = time.perf_counter() - wall0
    if ctx.dist is not None:
        ctx.dist.barrier()
    clocks = sampler.stop() if sampler else None
    launches = mlt.kernel_launches() - launches0
    mlt.sync_status(ctx.stream)
    total_ms = ctx.max_over_ranks(float(sum(s.elapsed_time(e) for s, e in zip(starts, ends))))
    return total_ms / steps, clocks, launches, wall


def phase_pass(ctx, step, steps):
    """Per-phase device times: a second pass of the same steps with the
    library's phase events on the same stream (kept out of the timed pass:
    events between kernels stop one kernel's launch from overlapping the
    previous kernel's tail)."""
    from paper_2411_10764_gb300 import mlt

    mlt.profile_phases(True)
    for i in range(steps):
        ctx.flush.fill_(float(i))
        step()
    phases, calls = mlt.phase_times()
    mlt.profile_phases(False)
    mlt.sync_status(ctx.stream)
    return {k: v / max(calls, 1) for k, v in phases.items()}


def walk_ceiling(ctx, w, model, x):
    """mlt_walk_peak on this batch: the same walk and layout over the first
    trees of `model` held in shared memory for the whole launch (no chunk
    streaming).  A decoded workload's first 2^22 candidates are materialised
    for it with mlt_decode_knobs."""
    import torch
    from paper_2411_10764_gb300 import mlt

    if model.depth > 10:
        return None
    mid = mlt.MLT_MODEL_V if model is w.v else mlt.MLT_MODEL_P
    if x is None:
        d = w.decoder
        _, x = mlt.decode_knobs(d.radices, d.option_values, d.program, w.first_index, min(w.n, 1 << 22),
                                device=ctx.dev, stream=ctx.stream)
    n = x.shape[0]
    _, visits1 = mlt.walk_peak(x, 1, model_id=mid, stream=ctx.stream)
    resident = visits1 // (n * model.depth)
    rounds = max(1, round(model.n_trees / resident))
    sums = None
    for _ in range(2):
        sums, _ = mlt.walk_peak(x, rounds, model_id=mid, out_sums=sums, stream=ctx.stream)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    reps = 5
    e0.record(ctx.stream)
    for _ in range(reps):
        _, visits = mlt.walk_peak(x, rounds, model_id=mid, out_sums=sums, stream=ctx.stream)
    e1.record(ctx.stream)
    torch.cuda.synchronize(ctx.dev)
    mlt.sync_status(ctx.stream)
    ms = e0.elapsed_time(e1) / reps
    return {"value": visits / (ms / 1e3) / 1e9, "unit": "Gvisit/s", "ms_per_launch": ms,
            "model": "V" if mid == mlt.MLT_MODEL_V else "P", "resident_trees": int(resident),
            "rounds": int(rounds), "rows": int(n),
            "what": "mlt_walk_peak: the same walk and layout over trees held in shared memory for the whole "
                    "launch (no chunk streaming)"}


def e2e_rate(ctx, w, step, bufs, steps):
    """The same metric through the host-buffer API: every step uploads its
    inputs from pinned host memory and downloads its results.  Returns
    (candidates/s over ranks, h2d bytes, d2h bytes, how, synchronous-call
    rate)."""
    import torch
    from paper_2411_10764_gb300 import mlt

    n, k, thr, d = w.n, w.k, w.thr, w.decoder
    hpv = torch.empty(n, dtype=torch.float32).pin_memory()
    hpf = torch.empty(n, dtype=torch.float32).pin_memory()
    htk = torch.empty(k, dtype=torch.int64).pin_memory()
    out = (hpv.numpy(), hpf.numpy(), htk.numpy())
    if d is None:
        hxn = torch.from_numpy(w.feats).pin_memory().numpy()
        h2d = int(w.feats.nbytes)

        def e2e_step():
            mlt.screen_host(hxn, thr, k, out=out, stream=ctx.stream)
    else:
        # a decoded workload's only input is its knob space (radices, option
        # values, feature program); its results are read back the same way
        h2d = int(d.radices.nbytes + d.option_values.nbytes + d.program.nbytes)

        def e2e_step():
            step()
            hpv.copy_(bufs["pv"], non_blocking=True)
            hpf.copy_(bufs["pf"], non_blocking=True)
            htk.copy_(bufs["tk"], non_blocking=True)
            ctx.stream.synchronize()
    for _ in range(3):
        e2e_step()
    t0 = time.perf_counter()
    for _ in range(steps):
        e2e_step()
    sync_s = (time.perf_counter() - t0) / steps
    best_s, how = sync_s, "mlt_screen_host: one synchronous call per batch"
    if d is None:
        # the pipelined entry point: every batch still uploads its features
        # and downloads its results, overlapped with the previous / next
        # batch's screening (two pinned result sets in turn)
        outs2 = [out, (torch.empty(n, dtype=torch.float32).pin_memory().numpy(),
                       torch.empty(n, dtype=torch.float32).pin_memory().numpy(),
                       torch.empty(k, dtype=torch.int64).pin_memory().numpy())]
        outs_b = [outs2[i & 1] for i in range(steps)]
        mlt.screen_host_batches([hxn] * 4, thr, k, outs=outs_b[:4], stream=ctx.stream)
        t0 = time.perf_counter()
        mlt.screen_host_batches([hxn] * steps, thr, k, outs=outs_b, stream=ctx.stream)
        pipe_s = (time.perf_counter() - t0) / steps
        if pipe_s < best_s:
            best_s = pipe_s
            how = (f"mlt_screen_host_batches: {steps} host batches in one call, each uploaded and downloaded, "
                   f"copies overlapped with screening")
    best_s = ctx.max_over_ranks(best_s)
    return ctx.world * n / best_s, h2d, int(2 * n * 4 + k * 8), how, ctx.world * n / sync_s


def measure_workload(ctx, w, args, headline: bool):
    """One workload's record: device-resident rate, phases, roofline
    fractions, near-decision counts, end-to-end rate, oracle baseline."""
    import torch
    from paper_2411_10764_gb300 import mlt

    mlt.load_workload_models(w)
    step, bufs = screen_step(ctx, w)
    for _ in range(max(3, args.warmup)):
        ctx.flush.fill_(1.0)
        step()
    mlt.sync_status(ctx.stream)
    survivors = mlt.last_survivor_count(ctx.stream)
    steps = args.steps
    if not headline:
        # enough steps for the clock samples (at least MIN_TIMED_S of work)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(ctx.stream)
        step()
        e1.record(ctx.stream)
        torch.cuda.synchronize(ctx.dev)
        est = max(e0.elapsed_time(e1), 1e-3)
        steps = int(min(20000, max(args.steps, math.ceil(MIN_TIMED_S * 1e3 / est))))
    jit0 = mlt.decode_jit_calls()
    ms, clocks, launches, wall = timed_steps(ctx, step, steps, ctx.rank == 0)
    jit_steps = mlt.decode_jit_calls() - jit0
    phases = phase_pass(ctx, step, min(steps, 200))
    pv, pf, tk = (bufs[k].cpu().numpy() for k in ("pv", "pf", "tk"))
    hbm_gbs, sm_max, peak_src = peaks()
    survived = None if w.cfg.shape == "full" else np.isfinite(pf[:2048])
    cnt = algorithmic_counts(w, survivors, survived)
    v_ms, p_ms = phases["v_pass"], phases["p_pass"]
    dominant = "v_pass" if v_ms >= p_ms else "p_pass"
    dom_ms = max(v_ms, p_ms)
    dom_visits = cnt["v_visits"] if dominant == "v_pass" else cnt["p_visits"]
    dom_model = w.v if dominant == "v_pass" else w.p
    # one shared-memory gather of x[feature] per node visit, 32 lanes per
    # clock per SM: the on-chip issue ceiling of the walk
    visit_peak = SM_COUNT * 32 * sm_max * 1e6
    achieved = dom_visits / (dom_ms / 1e3)
    dom_bytes = (cnt["feat_bytes"] + cnt["v_table_bytes"]) if dominant == "v_pass" else \
        (cnt["survivor_feat_bytes"] + cnt["p_table_bytes"])
    step_bytes = cnt["feat_bytes"] + cnt["v_table_bytes"] + cnt["p_table_bytes"]
    ceiling = walk_ceiling(ctx, w, dom_model, bufs["x"]) if ctx.world == 1 else None
    value = ctx.world * w.n / (ms / 1e3)
    e2e_steps = max(10, min(args.steps, 200 if w.n <= (1 << 20) else 10))
    e2e_v, h2d, d2h, how, sync_v = e2e_rate(ctx, w, step, bufs, e2e_steps)
    rec = {
        "workload": f"{w.cfg.name} (workload {w.cfg.id})", "n": w.n,
        "value": value, "unit": "candidates/s", "ms_per_step": ms, "steps": steps,
        "survivors": survivors, "survivor_rate": survivors / max(w.n, 1),
        "phases_ms": phases,
        "phases_note": "second pass of the same steps with CUDA events between phases",
        "roofline": {
            "bound": "alu", "kernel": f"{dominant} (tree walk)",
            "achieved": achieved / 1e9, "peak": visit_peak / 1e9, "unit": "Gvisit/s",
            "frac": achieved / visit_peak,
            # the committed counters were taken at each workload's full size
            "traffic": dram_traffic(w.cfg.id, dominant) if w.n == w.cfg.n else None,
            "peak_note": f"152 SMs x 32 shared-memory lanes/clk x {sm_max:.0f} MHz: one x[f] gather per node visit",
            "measured_walk_peak": None if ceiling is None else dict(ceiling, frac=achieved / 1e9 / ceiling["value"]),
        },
        "hbm_roofline": {
            "bound": "hbm", "achieved": step_bytes / (ms / 1e3) / 1e9, "peak": hbm_gbs,
            "unit": "GB/s", "frac": step_bytes / (ms / 1e3) / 1e9 / hbm_gbs,
            "peak_source": peak_src, "bytes_per_step": step_bytes,
            "frac_of_nominal_7900": step_bytes / (ms / 1e3) / 1e9 / 7900.0,
            "dominant_kernel_gbs": dom_bytes / (dom_ms / 1e3) / 1e9,
            "dominant_kernel_frac": dom_bytes / (dom_ms / 1e3) / 1e9 / hbm_gbs,
            "target": "0.60 of the HBM roofline on workloads 2-4: not reached (the walk is bound on chip, "
                      "not by HBM; see roofline)",
        },
        "near_decisions": near_counts(pv, pf, tk, w.thr, w.first_index),
        "e2e": {"value": e2e_v, "unit": "candidates/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "how": how, "sync_call_value": sync_v},
        "gpu_launches": int(launches), "clocks": clocks,
        "wall_ms_per_step_incl_flush": wall * 1e3 / steps,
    }
    rec["walk_shapes"] = {"v": mlt.walk_shape(mlt.MLT_MODEL_V, w.n), "p": mlt.walk_shape(mlt.MLT_MODEL_P, w.n, True),
                          "note": "planned shape of each pass's walk (a step of one launch uses the single-launch "
                                  "kernel instead)" if launches == steps else "planned shape of each pass's walk"}
    if w.decoder is not None:
        rec["decode_path"] = ("compiled feature program (NVRTC): rows written once per step, then screened"
                              if jit_steps == steps else "interpreted inside the walk kernels")
    if ctx.rank == 0 and ctx.world == 1 and not args.no_cpu_baseline:
        rec["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds if headline else args.cpu_seconds_per_config)
    return rec, bufs


def next_rows(ctx, w2, seed, args):
    """The rows after the screening step, each timed on the workload it
    applies to: model A's rerank, the half-table variant and the batched
    accumulation on the gemm batch (stored features); the explorer's
    proposal step and the knob decoder on the conv2d knob space."""
    import torch
    from paper_2411_10764_gb300 import mlt
    from paper_2411_10764_gb300 import workloads as W

    out = {}
    dev, stream = ctx.dev, ctx.stream
    mlt.load_workload_models(w2)
    step, bufs = screen_step(ctx, w2)
    x, pf, tk = bufs["x"], bufs["pf"], bufs["tk"]
    n, k, thr = w2.n, w2.k, w2.thr
    for _ in range(3):
        step()
    mlt.sync_status(stream)
    survivors = mlt.last_survivor_count(stream)
    # model A's rerank of the kept (alpha+1)N = k candidates down to N = k/2
    # (alpha = 1): 300 trees, depth <= 14 (Table 3)
    a = W.make_model_a(w2, seed=seed)
    mlt.load_ensemble(mlt.MLT_MODEL_A, a.nodes, a.n_trees, a.depth)
    n_final = max(1, k // 2)
    sc = torch.empty(k, dtype=torch.float32, device=dev)
    fin = torch.empty(n_final, dtype=torch.int64, device=dev)
    for _ in range(5):
        mlt.rerank(x, tk, n_final, sc, fin, stream=stream)
    reps = 50
    r0 = torch.cuda.Event(enable_timing=True)
    r1 = torch.cuda.Event(enable_timing=True)
    r0.record(stream)
    for _ in range(reps):
        mlt.rerank(x, tk, n_final, sc, fin, stream=stream)
    r1.record(stream)
    torch.cuda.synchronize(dev)
    mlt.sync_status(stream)
    out["rerank"] = {"what": f"model A rerank of the top-{k} of {w2.cfg.name} to {n_final}", "a_trees": a.n_trees,
                     "a_max_depth": a.depth, "a_nodes": int((a.nodes["feature"] != -2).sum()),
                     "us_per_call": r0.elapsed_time(r1) * 1e3 / reps}

    # the half-table variant (binary16 thresholds, leaves and staged
    # features): it changes results, so its agreement with the fp32 run is
    # reported beside its speed
    ref_valid = torch.isfinite(pf).cpu().numpy()
    ref_topk = tk.cpu().numpy()
    mlt.load_workload_models(w2, half=True)
    for _ in range(3):
        ctx.flush.fill_(1.0)
        step()
    h_steps = max(10, min(args.steps * 25, 500))
    h_ms, _, _, _ = timed_steps(ctx, step, h_steps, False)
    h_phases = phase_pass(ctx, step, min(h_steps, 50))
    out["half_tables"] = {
        "workload": w2.cfg.name, "value": n / (h_ms / 1e3), "unit": "candidates/s", "ms_per_step": h_ms,
        "steps": h_steps, "phases_ms": h_phases,
        "decision_agreement": float((torch.isfinite(pf).cpu().numpy() == ref_valid).mean()),
        "topk_overlap": len(set(tk.cpu().numpy().tolist()) & set(ref_topk.tolist())) / k,
        "what": "mlt_load_ensemble_f16: binary16 thresholds, leaves and staged features; changes results "
                "(parity is against the rounded model); agreement and top-k overlap are against the fp32 run"}
    mlt.load_workload_models(w2)

    # batched accumulation (mlt_screen_until) on the same batch
    target = max(k, survivors // 4)
    batch = max(32, n // 8)
    for _ in range(3):
        mlt.screen_until(x, batch, target, thr, k, stream=stream)
    a0 = torch.cuda.Event(enable_timing=True)
    a1 = torch.cuda.Event(enable_timing=True)
    reps = 20
    a0.record(stream)
    for _ in range(reps):
        _, _, _, st_ = mlt.screen_until(x, batch, target, thr, k, stream=stream)
    a1.record(stream)
    torch.cuda.synchronize(dev)
    mlt.sync_status(stream)
    consumed, kept, batches = (int(v) for v in st_.cpu().tolist())
    acc_ms = a0.elapsed_time(a1) / reps
    out["accumulation"] = {"what": f"mlt_screen_until on {w2.cfg.name}: batches of {batch}, stop once {target} "
                                   f"valid candidates are kept",
                           "ms_per_call": acc_ms, "consumed": consumed, "kept": kept, "batches": batches,
                           "candidates_per_s": consumed / (acc_ms / 1e3)}
    del step, bufs, x, pf, tk

    # the explorer's proposal step (mlt_sa_step) and the knob decoder over
    # the conv2d knob space
    w4 = W.make_workload(4, seed=seed, n=1)
    mlt.load_workload_models(w4)
    dec4 = w4.decoder
    m_chains = 1 << 20
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    parent = torch.randint(0, dec4.space, (m_chains,), device=dev, dtype=torch.int64, generator=gen)
    pscore = torch.full((m_chains,), float("-inf"), device=dev)
    s_steps = 10
    draws = [(torch.randint(0, 1 << 30, (m_chains,), device=dev, dtype=torch.int32, generator=gen),
              torch.randint(0, 1 << 30, (m_chains,), device=dev, dtype=torch.int32, generator=gen),
              torch.log(torch.rand(m_chains, device=dev, generator=gen)))
             for _ in range(s_steps + 2)]
    for i in range(2):
        parent, pscore, _ = mlt.sa_step(dec4.radices, dec4.option_values, dec4.program, parent, pscore,
                                        *draws[i], 1.0, w4.thr, stream=stream)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(2, s_steps + 2):
        parent, pscore, acc_ = mlt.sa_step(dec4.radices, dec4.option_values, dec4.program, parent, pscore,
                                           *draws[i], 1.0, w4.thr, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    mlt.sync_status(stream)
    sa_ms = e0.elapsed_time(e1) / s_steps
    out["sa_step"] = {"what": f"mlt_sa_step: {m_chains} simulated-annealing chains over the conv2d knob space "
                              f"(decode, V {w4.v.n_trees}x d{w4.v.depth}, P {w4.p.n_trees}x d{w4.p.depth}, "
                              f"Metropolis at T=1)",
                      "ms_per_step": sa_ms, "proposals_per_s": m_chains / (sa_ms / 1e3),
                      "accepted_last_step": int(acc_.sum().item()) / m_chains}
    # the knob decoder on its own (mlt_decode_knobs): 2^22 candidates
    # materialised as option indices and features, an HBM write stream
    n_dec = 1 << 22
    for _ in range(2):
        mlt.decode_knobs(dec4.radices, dec4.option_values, dec4.program, 0, n_dec, device=dev, stream=stream)
    torch.cuda.synchronize(dev)
    reps = 10
    e0.record(stream)
    for i in range(reps):
        kn, fe = mlt.decode_knobs(dec4.radices, dec4.option_values, dec4.program, (i % 4) * n_dec, n_dec,
                                  device=dev, stream=stream)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    mlt.sync_status(stream)
    dec_ms = e0.elapsed_time(e1) / reps
    dec_bytes = kn.numel() * kn.element_size() + fe.numel() * fe.element_size()
    out["decode_knobs"] = {"what": f"mlt_decode_knobs: {n_dec} conv2d candidates to {dec4.radices.size} option "
                                   f"indices (u8) and {dec4.program.size} fp32 features each",
                           "ms_per_call": dec_ms, "candidates_per_s": n_dec / (dec_ms / 1e3),
                           "bytes_written": int(dec_bytes), "write_gbs": dec_bytes / (dec_ms / 1e3) / 1e9}
    return out


def run_ours(args):
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)

    from paper_2411_10764_gb300 import workloads as W

    ctx = Ctx(dev, torch.cuda.current_stream(dev), world, rank, dist)
    seed = args.seed + rank
    w = W.make_workload(args.workload, seed=seed, n=args.n)
    head, head_bufs = measure_workload(ctx, w, args, headline=True)
    del head_bufs
    torch.cuda.empty_cache()

    per_config = None
    extra = None
    if world == 1 and not args.no_per_config:
        per_config = {}
        for wid in ALL_WORKLOADS:
            if wid == args.workload and args.n is None:
                per_config[str(wid)] = {kk: vv for kk, vv in head.items()}
                continue
            wc = W.make_workload(wid, seed=seed)
            rec, bufs = measure_workload(ctx, wc, args, headline=False)
            per_config[str(wid)] = rec
            del bufs, wc
            torch.cuda.empty_cache()
    if world == 1 and not args.no_next:
        extra = next_rows(ctx, W.make_workload(2, seed=seed), seed, args)
        torch.cuda.empty_cache()

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0
    line = {
        "metric": METRIC, "value": head["value"], "unit": "candidates/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded; shapes of the paper's tuning tasks)",
        "config": config_dict(w, args.seed, world),
        "survivors": head["survivors"],
        "phases_ms": head["phases_ms"], "phases_note": head["phases_note"],
        "roofline": head["roofline"], "hbm_roofline": head["hbm_roofline"],
        "near_decisions": head["near_decisions"],
        "e2e": head["e2e"], "gpu_launches": head["gpu_launches"], "clocks": head["clocks"],
        "wall_ms_per_step_incl_flush": head["wall_ms_per_step_incl_flush"],
    }
    if "cpu_baseline" in head:
        line["cpu_baseline"] = head["cpu_baseline"]
    if "decode_path" in head:
        line["decode_path"] = head["decode_path"]
    line["walk_shapes"] = head["walk_shapes"]
    if per_config is not None:
        line["per_config"] = per_config
    if extra is not None:
        line["next_rows"] = extra
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", type=int, default=DEFAULT_WORKLOAD,
                    help="headline workload 1-5 (1 tiny, 2 gemm, 3 sa-batch, 4 conv2d decoded, 5 skewed-nan)")
    ap.add_argument("--seed", type=int, default=1)
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="oracle time for the headline workload's CPU baseline")
    ap.add_argument("--cpu-seconds-per-config", type=float, default=4.0,
                    help="oracle time for each other workload's CPU baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="only the headline workload (no per-workload records)")
    ap.add_argument("--no-next", action="store_true",
                    help="skip the rerank, half-table, accumulation, explorer-step and decoder timings")
    ap.add_argument("--no-rerank", action="store_true", help=argparse.SUPPRESS)  # older command lines:
    ap.add_argument("--no-half", action="store_true", help=argparse.SUPPRESS)    # same as --no-next
    ap.add_argument("--n", type=int, default=None,
                    help="candidates per batch (default: the workload's size; smaller for profiling captures)")
    args = ap.parse_args()
    args.no_next = args.no_next or args.no_rerank or args.no_half
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
