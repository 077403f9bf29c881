"""Benchmark: candidates screened per second (V filter + P score + top-k) on
GB300, with roofline, CPU-oracle baseline and end-to-end figures.

One step = one mlt_screen call over one batch of the "GEMM-style schedule
space" workload: 65,536 candidates x 64 fp32 features, V = 200 trees of
depth 8, P = 400 trees of depth 8, validity threshold 0.5, top-128 (the
batch shape of ML^2Tuner's explorer step, Sec. 2; tree ensembles as in
Table 3).  The inputs sit in HBM before the timed region; L2 is flushed
(a 256 MB device write) before every timed step, outside its events.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun every rank screens its own batch (different seed): weak
scaling, no collective on the data path; rank 0 prints the JSON line with
the max-over-ranks time.  `--impl reference` times the CPU oracle instead
(rank 0 only).
"""
from __future__ import annotations

import argparse
import json
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
DEFAULT_WORKLOAD = 2
L2_FLUSH_BYTES = 256 << 20
SM_COUNT = 152
SM_MAX_MHZ_NOMINAL = 2070.0


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p.get("sm_max_mhz", SM_MAX_MHZ_NOMINAL)), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, SM_MAX_MHZ_NOMINAL, "fallback"


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


def oracle_rate(w, budget_s: float, rows_per_call: int | None = None):
    """Single-threaded oracle throughput (candidates/s) on leading rows of
    the workload: whole oracle passes (screen + top-k) of `rows_per_call`
    rows until `budget_s` seconds have been spent."""
    if rows_per_call is None:
        # whole workload if one pass fits the budget, else a leading slice
        probe = min(w.n, 1024)
        t0 = time.perf_counter()
        oracle_pass(w, probe)
        per_row = (time.perf_counter() - t0) / probe
        rows_per_call = int(max(probe, budget_s / 4 / max(per_row, 1e-9)))
    n = min(w.n, rows_per_call)
    done, t0 = 0, time.perf_counter()
    calls = 0
    while True:
        oracle_pass(w, n)
        done += n
        calls += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            break
    return done / el, {"rows_per_call": n, "calls": calls, "seconds": round(el, 3)}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
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
    sample = f"first {rows} of {w.n} candidates per step (whole oracle pass: {what})"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "candidates/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": mean * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": config_dict(w),
        "cpu_baseline": {"value": value, "unit": "candidates/s", "cores": 1, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "candidates/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def config_dict(w):
    c = w.cfg
    return {"workload": f"{c.name} (workload {c.id})", "n": w.n, "F": c.F,
            "v_trees": c.v_trees, "v_depth": c.v_depth, "p_trees": c.p_trees, "p_depth": c.p_depth,
            "thr": c.thr, "k": c.k, "seed": None,
            "l2": "flushed before every timed step (256 MB device write, outside the step events)"}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
def walk_source_hash() -> str:
    """Hash of the sources the tree-walk kernels compile from (the walk
    device code, the launch planners and instantiations, the internal
    header), in a fixed order."""
    import glob
    import hashlib

    csrc = os.path.join(ROOT, "paper_2411_10764_gb300", "csrc")
    files = [os.path.join(csrc, "walk.cuh"), os.path.join(csrc, "mlt_internal.cuh")]
    files += sorted(glob.glob(os.path.join(csrc, "traverse*.cu")))
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
    """Node visits and algorithmic HBM bytes of one step (see the design
    notes).  Full trees: trees x depth visits per candidate; unbalanced
    trees: trees x the mean path length over a 2,048-row sample (the P
    pass's over the sample's survivors)."""
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
    # 8 B per split node (threshold + feature), 4 B per leaf value
    def table(ens):
        f = ens.nodes["feature"]
        return int((f >= 0).sum()) * 8 + int((f == -1).sum()) * 4

    v_table, p_table = table(w.v), table(w.p)
    out_bytes = w.n * 8 + c.k * 8
    return {"v_visits": v_visits, "p_visits": p_visits, "v_path": v_path, "p_path": p_path,
            "feat_bytes": feat_bytes,
            "v_table_bytes": v_table, "p_table_bytes": p_table, "out_bytes": out_bytes,
            "survivor_feat_bytes": survivors * c.F * 4}


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

    from paper_2411_10764_gb300 import mlt
    from paper_2411_10764_gb300 import workloads as W

    seed = args.seed + rank
    w = W.make_workload(args.workload, seed=seed, n=args.n)
    mlt.load_workload_models(w)
    n, k, thr = w.n, w.k, w.thr
    pv = torch.empty(n, dtype=torch.float32, device=dev)
    pf = torch.empty(n, dtype=torch.float32, device=dev)
    tk = torch.empty(k, dtype=torch.int64, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    d = w.decoder
    x = None if d is not None else torch.from_numpy(w.feats).to(dev)

    def step():
        if d is None:
            mlt.screen(x, thr, k, pv, pf, tk, stream=stream)
        else:
            # knob indices decoded and featurised inside the walk kernels
            mlt.screen_decoded(d.radices, d.option_values, d.program, w.first_index, n, thr, k,
                               out_pvalid=pv, out_perf=pf, out_topk=tk, stream=stream)

    for _ in range(max(3, args.warmup)):
        flush.fill_(1.0)
        step()
    mlt.sync_status(stream)
    survivors = mlt.last_survivor_count(stream)

    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid) if rank == 0 else None

    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize(dev)
    if sampler:
        sampler.start()
    launches0 = mlt.kernel_launches()
    wall0 = time.perf_counter()
    for i in range(args.steps):
        flush.fill_(float(i))
        starts[i].record(stream)
        step()
        ends[i].record(stream)
    torch.cuda.synchronize(dev)
    wall = time.perf_counter() - wall0
    if dist is not None:
        dist.barrier()
    clocks = sampler.stop() if sampler else None
    launches = mlt.kernel_launches() - launches0
    mlt.sync_status(stream)
    # per-phase device times: a second pass of the same steps with the
    # library's phase events on the same stream (kept out of the timed pass:
    # events between kernels stop one kernel's launch from overlapping the
    # previous kernel's tail)
    mlt.profile_phases(True)
    for i in range(args.steps):
        flush.fill_(float(i))
        step()
    phases, calls = mlt.phase_times()
    mlt.profile_phases(False)
    mlt.sync_status(stream)
    step_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    total_ms = float(sum(step_ms))
    if dist is not None:
        t = torch.tensor([total_ms], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_per_step = total_ms / args.steps
    value = world * n / (ms_per_step / 1e3)

    # model A's rerank of the kept (alpha+1)N = k candidates down to N = k/2
    # (alpha = 1): 300 trees, depth <= 14 (Table 3), timed per call
    rerank = None
    if not args.no_rerank and x is not None:
        a = W.make_model_a(w, seed=seed)
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
        nodes_a = int((a.nodes["feature"] != -2).sum())
        rerank = {"what": f"model A rerank of the top-{k} to {n_final}", "a_trees": a.n_trees,
                  "a_max_depth": a.depth, "a_nodes": nodes_a, "us_per_call": r0.elapsed_time(r1) * 1e3 / reps}

    # end to end through the host-buffer entry point (pinned host memory);
    # a decoded workload's only input is its knob space (radices, option
    # values, feature program), and its results are read back the same way
    hpv = torch.empty(n, dtype=torch.float32).pin_memory()
    hpf = torch.empty(n, dtype=torch.float32).pin_memory()
    htk = torch.empty(k, dtype=torch.int64).pin_memory()
    out = (hpv.numpy(), hpf.numpy(), htk.numpy())
    if d is None:
        hxn = torch.from_numpy(w.feats).pin_memory().numpy()
        h2d_bytes = int(w.feats.nbytes)

        def e2e_step():
            mlt.screen_host(hxn, thr, k, out=out, stream=stream)
    else:
        h2d_bytes = int(d.radices.nbytes + d.option_values.nbytes + d.program.nbytes)

        def e2e_step():
            step()
            hpv.copy_(pv, non_blocking=True)
            hpf.copy_(pf, non_blocking=True)
            htk.copy_(tk, non_blocking=True)
            torch.cuda.current_stream(dev).synchronize()
    for _ in range(3):
        e2e_step()
    e2e_steps = max(10, min(args.steps, 200 if n <= (1 << 20) else 10))
    # one synchronous call per batch (upload, screen, download in turn)
    t0 = time.perf_counter()
    for _ in range(e2e_steps):
        e2e_step()
    e2e_sync_s = (time.perf_counter() - t0) / e2e_steps
    e2e_s = e2e_sync_s
    e2e_how = "mlt_screen_host: one synchronous call per batch"
    if d is None:
        # the pipelined entry point: every batch still uploads its features
        # and downloads its results, overlapped with the previous / next
        # batch's screening (two pinned result sets in turn)
        outs2 = [out, (torch.empty(n, dtype=torch.float32).pin_memory().numpy(),
                       torch.empty(n, dtype=torch.float32).pin_memory().numpy(),
                       torch.empty(k, dtype=torch.int64).pin_memory().numpy())]
        outs_b = [outs2[i & 1] for i in range(e2e_steps)]
        mlt.screen_host_batches([hxn] * 4, thr, k, outs=outs_b[:4], stream=stream)
        t0 = time.perf_counter()
        mlt.screen_host_batches([hxn] * e2e_steps, thr, k, outs=outs_b, stream=stream)
        pipe_s = (time.perf_counter() - t0) / e2e_steps
        if pipe_s < e2e_s:
            e2e_s = pipe_s
            e2e_how = (f"mlt_screen_host_batches: {e2e_steps} host batches in one call, each uploaded and "
                       f"downloaded, copies overlapped with screening")
    if dist is not None:
        t = torch.tensor([e2e_s], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        e2e_s = float(t.item())

    # the half-table variant (binary16 thresholds, leaves and staged
    # features): same batch, same timing protocol; it changes results, so
    # its agreement with the fp32 run is reported beside its speed
    half = None
    if not args.no_half and d is None and max(w.v.depth, w.p.depth) <= 10:
        ref_valid = torch.isfinite(pf).cpu().numpy()
        ref_topk = tk.cpu().numpy()
        mlt.load_workload_models(w, half=True)
        for _ in range(max(3, args.warmup)):
            flush.fill_(1.0)
            step()
        h_steps = max(10, min(args.steps, 500))
        hs = [torch.cuda.Event(enable_timing=True) for _ in range(h_steps)]
        he = [torch.cuda.Event(enable_timing=True) for _ in range(h_steps)]
        torch.cuda.synchronize(dev)
        for i in range(h_steps):
            flush.fill_(float(i))
            hs[i].record(stream)
            step()
            he[i].record(stream)
        torch.cuda.synchronize(dev)
        mlt.sync_status(stream)
        h_ms = float(sum(a.elapsed_time(b) for a, b in zip(hs, he))) / h_steps
        mlt.profile_phases(True)
        for i in range(min(h_steps, 50)):
            flush.fill_(float(i))
            step()
        h_phases, h_calls = mlt.phase_times()
        mlt.profile_phases(False)
        h_valid = torch.isfinite(pf).cpu().numpy()
        h_topk = tk.cpu().numpy()
        half = {"value": world * n / (h_ms / 1e3), "unit": "candidates/s", "ms_per_step": h_ms,
                "steps": h_steps,
                "phases_ms": {kk: vv / max(h_calls, 1) for kk, vv in h_phases.items()},
                "decision_agreement": float((h_valid == ref_valid).mean()),
                "topk_overlap": len(set(h_topk.tolist()) & set(ref_topk.tolist())) / k,
                "what": "mlt_load_ensemble_f16: binary16 thresholds, leaves and staged features; "
                        "changes results (parity is against the rounded model); agreement and top-k "
                        "overlap are against the fp32 run on the same batch"}
        mlt.load_workload_models(w)

    # the next rows of the path: batched accumulation (mlt_screen_until) on
    # this batch, and the explorer's proposal step (mlt_sa_step) over the
    # decoded conv2d knob space
    accumulation = sa = decode = None
    if not args.no_next and d is None:
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
        accumulation = {"what": f"mlt_screen_until: batches of {batch}, stop once {target} valid candidates are kept",
                        "ms_per_call": acc_ms, "consumed": consumed, "kept": kept, "batches": batches,
                        "candidates_per_s": consumed / (acc_ms / 1e3)}
    if not args.no_next:
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
        accepted = 0
        for i in range(2, s_steps + 2):
            parent, pscore, acc_ = mlt.sa_step(dec4.radices, dec4.option_values, dec4.program, parent, pscore,
                                               *draws[i], 1.0, w4.thr, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        mlt.sync_status(stream)
        accepted = int(acc_.sum().item())
        sa_ms = e0.elapsed_time(e1) / s_steps
        sa = {"what": f"mlt_sa_step: {m_chains} simulated-annealing chains over the conv2d knob space "
                      f"(decode, V {w4.v.n_trees}x d{w4.v.depth}, P {w4.p.n_trees}x d{w4.p.depth}, Metropolis at T=1)",
              "ms_per_step": sa_ms, "proposals_per_s": m_chains / (sa_ms / 1e3),
              "accepted_last_step": accepted / m_chains}
        # the knob decoder on its own (mlt_decode_knobs): 2^22 candidates of
        # the same space materialised as option indices and features, an HBM
        # write stream
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
        decode = {"what": f"mlt_decode_knobs: {n_dec} conv2d candidates to {dec4.radices.size} option indices "
                          f"(u8) and {dec4.program.size} fp32 features each",
                  "ms_per_call": dec_ms, "candidates_per_s": n_dec / (dec_ms / 1e3),
                  "bytes_written": int(dec_bytes), "write_gbs": dec_bytes / (dec_ms / 1e3) / 1e9}
        mlt.load_workload_models(w)

    # the walk-rate ceiling of the dominant pass's model on this batch
    # (mlt_walk_peak): the same walk over trees held in shared memory for
    # the whole launch, no chunk streaming
    walk_peak = None
    v_ms0 = phases["v_pass"] / max(calls, 1)
    p_ms0 = phases["p_pass"] / max(calls, 1)
    peak_model = w.v if v_ms0 >= p_ms0 else w.p
    if d is None and peak_model.depth <= 10:
        mid = mlt.MLT_MODEL_V if peak_model is w.v else mlt.MLT_MODEL_P
        _, visits1 = mlt.walk_peak(x, 1, model_id=mid, stream=stream)
        resident = visits1 // (n * peak_model.depth)
        rounds = max(1, round(peak_model.n_trees / resident))
        sums = None
        for _ in range(2):
            sums, _ = mlt.walk_peak(x, rounds, model_id=mid, out_sums=sums, stream=stream)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        reps = 5
        e0.record(stream)
        for _ in range(reps):
            _, visits = mlt.walk_peak(x, rounds, model_id=mid, out_sums=sums, stream=stream)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        mlt.sync_status(stream)
        wp_ms = e0.elapsed_time(e1) / reps
        walk_peak = {"value": visits / (wp_ms / 1e3) / 1e9, "unit": "Gvisit/s", "ms_per_launch": wp_ms,
                     "model": "V" if mid == mlt.MLT_MODEL_V else "P", "resident_trees": int(resident),
                     "rounds": int(rounds),
                     "what": "mlt_walk_peak: the same walk and layout over trees held in shared memory for "
                             "the whole launch (no chunk streaming), every row of the batch"}

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return 0

    hbm_gbs, sm_max, peak_src = peaks()
    survived = None
    if w.cfg.shape != "full":
        survived = torch.isfinite(pf[:2048]).cpu().numpy()
    cnt = algorithmic_counts(w, survivors, survived)
    v_ms = phases["v_pass"] / max(calls, 1)
    p_ms = phases["p_pass"] / max(calls, 1)
    dominant = "v_pass" if v_ms >= p_ms else "p_pass"
    dom_ms = max(v_ms, p_ms)
    dom_visits = cnt["v_visits"] if dominant == "v_pass" else cnt["p_visits"]
    # one shared-memory gather of x[feature] per node visit, 32 lanes per
    # clock per SM: the on-chip issue ceiling of the walk
    visit_peak = SM_COUNT * 32 * sm_max * 1e6
    achieved = dom_visits / (dom_ms / 1e3)
    dom_bytes = (cnt["feat_bytes"] + cnt["v_table_bytes"]) if dominant == "v_pass" else \
        (cnt["survivor_feat_bytes"] + cnt["p_table_bytes"])
    step_bytes = cnt["feat_bytes"] + cnt["v_table_bytes"] + cnt["p_table_bytes"]
    traffic = dram_traffic(args.workload, dominant)
    line = {
        "metric": METRIC, "value": value, "unit": "candidates/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded; shapes of the paper's tuning tasks)",
        "config": dict(config_dict(w), seed=args.seed, parallelism=f"replicas x{world}"),
        "survivors": survivors,
        "phases_ms": {kk: vv / max(calls, 1) for kk, vv in phases.items()},
        "phases_note": "second pass of the same steps with CUDA events between phases",
        "roofline": {
            "bound": "alu", "kernel": f"{dominant} (tree walk)",
            "achieved": achieved / 1e9, "peak": visit_peak / 1e9, "unit": "Gvisit/s",
            "frac": achieved / visit_peak, "traffic": traffic,
            "peak_note": f"152 SMs x 32 shared-memory lanes/clk x {sm_max:.0f} MHz: one x[f] gather per node visit",
            "measured_walk_peak": None if walk_peak is None else dict(
                walk_peak, frac=achieved / 1e9 / walk_peak["value"]),
        },
        "hbm_roofline": {
            "bound": "hbm", "achieved": step_bytes / (ms_per_step / 1e3) / 1e9, "peak": hbm_gbs,
            "unit": "GB/s", "frac": step_bytes / (ms_per_step / 1e3) / 1e9 / hbm_gbs,
            "peak_source": peak_src, "bytes_per_step": step_bytes,
            "frac_of_nominal_7900": step_bytes / (ms_per_step / 1e3) / 1e9 / 7900.0,
            "dominant_kernel_gbs": dom_bytes / (dom_ms / 1e3) / 1e9,
        },
        "e2e": {"value": world * n / e2e_s, "unit": "candidates/s",
                "h2d_bytes_per_step": h2d_bytes,
                "d2h_bytes_per_step": int(2 * n * 4 + k * 8),
                "how": e2e_how, "sync_call_value": world * n / e2e_sync_s},
        "gpu_launches": int(launches),
        "rerank": rerank,
        "half_tables": half,
        "accumulation": accumulation,
        "sa_step": sa,
        "decode_knobs": decode,
        "clocks": clocks,
        "wall_ms_per_step_incl_flush": wall * 1e3 / args.steps,
    }
    if not args.no_cpu_baseline:
        rate, info = oracle_rate(w, args.cpu_seconds)
        line["cpu_baseline"] = {"value": rate, "unit": "candidates/s", "cores": 1, "kind": "oracle",
                                "sample": f"first {info['rows_per_call']} of {w.n} candidates x "
                                          f"{info['calls']} oracle passes, {info['seconds']} s, single thread"}
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", type=int, default=DEFAULT_WORKLOAD,
                    help="workload 1-5 (1 tiny, 2 gemm, 3 sa-batch, 4 conv2d decoded, 5 skewed-nan)")
    ap.add_argument("--seed", type=int, default=1)
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-rerank", action="store_true")
    ap.add_argument("--no-half", action="store_true", help="skip the half-table variant's timing")
    ap.add_argument("--no-next", action="store_true",
                    help="skip the accumulation and explorer-step timings")
    ap.add_argument("--n", type=int, default=None,
                    help="candidates per batch (default: the workload's size; smaller for profiling captures)")
    args = ap.parse_args()
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
