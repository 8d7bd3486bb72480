#!/usr/bin/env python
"""Benchmark of the TokenTiming verification step on GB300.

One step = one tt_step over a batch: DTW alignment of every request, one pass
over the mapped draft rows and all target rows, and the per-request
accept / residual-sampling decision. Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle, timed on the host

Under torchrun every rank runs its own batch (requests are independent; no
collective on the data path) and the timed region is bracketed by barriers;
the reported time is the maximum over ranks (weak scaling).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "b1024_g8_v201k_bf16"
METRIC = "verified draft positions/sec (batch×γ) and HBM GB/s vs 8 TB/s; DTW pairs/sec"
UNIT = "positions/s"
L2_BYTES = 129 * 1024 * 1024
FALLBACK_HBM_GBS = 6800.0
ROWPASS_SOURCES = ["paper_2510_15545_gb300/csrc/rowpass.cu",
                   "paper_2510_15545_gb300/csrc/tt_device.cuh",
                   "paper_2510_15545_gb300/csrc/tt_launch.h"]


def parse_args(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["mine", "reference"], default="mine")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--batch", type=int, default=None,
                    help="requests per GPU (default: the workload's own batch); smaller "
                         "batches are for profiler captures, not bench lines")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="time only --workload, not also the other workloads")
    ap.add_argument("--temp", type=float, default=None,
                    help="temperature of draft and target rows (default: the workload's)")
    ap.add_argument("--top-k", type=int, default=0,
                    help="top-k filter of draft and target rows (0 = off)")
    ap.add_argument("--top-p", type=float, default=1.0,
                    help="top-p filter (after the top-k when --top-k is set; over the whole row "
                         "when it is not; 1 = off)")
    ap.add_argument("--rep-penalty", type=float, default=1.0,
                    help="repetition penalty of draft and target rows (1 = off; needs --top-k); "
                         "each request gets a seeded history of 64-1024 earlier tokens per family")
    ap.add_argument("--shards", type=int, default=0,
                    help="also time the vocabulary-sharded verification with the target "
                         "rows split into this many column slices (1-8), against the "
                         "unsplit verification (outside the timed region)")
    ap.add_argument("--no-reencode", action="store_true",
                    help="skip timing the re-encoding, Lemma-1 check and delta-pos histogram")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="CPU work budget of the oracle baseline sample")
    return ap.parse_args(argv)


# ----------------------------------------------------------- multi-process

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, ws, local


def dist_init(ws, backend):
    import torch.distributed as dist
    if ws > 1 and not dist.is_initialized():
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group(backend=backend)


def request_base(rank: int, batch: int) -> int:
    """Global index of a rank's first request: ranks own disjoint Philox streams."""
    return rank * batch


def barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(value: float, ws: int, device=None) -> float:
    """Largest value over ranks (the slowest rank sets the job's time)."""
    if ws <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(value: float, ws: int, device=None) -> float:
    if ws <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64,
                     device=device if device is not None else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


# ------------------------------------------------------------------ clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons, kept with host
    timestamps so that only the samples inside the timed region count."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, period_ms: int = 50):
        self.samples = []
        self.proc = None
        self.thread = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-i", str(gpu_index), "-lms", str(period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.perf_counter(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float) -> dict:
        inside = [s for t, s in self.samples if t0 <= t <= t1]
        note = "samples inside the timed region"
        if not inside and self.samples:  # a very short region: nearest samples
            inside = [min(self.samples, key=lambda ts: abs(ts[0] - 0.5 * (t0 + t1)))[1]]
            note = "nearest sample to a timed region shorter than the sampling period"
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for s in inside:
            try:
                sm.append(float(s[1]))
                smax.append(float(s[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, s[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": sorted(reasons),
                "samples": len(inside), "note": note}


# ----------------------------------------------------------------- helpers

def measured_hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def rowpass_source_hash() -> str:
    h = hashlib.sha256()
    for rel in ROWPASS_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, top_k: int = 0):
    """DRAM bytes per row-pass launch from the committed ncu summary, if it was
    taken on the current row-pass source (and, with filters, at the same top_k:
    the lists the pass writes are top_k entries per unit)."""
    name = "rowpass_filtered_%s.md" if top_k > 0 else "rowpass_%s.md"
    path = os.path.join(ROOT, "profiles", name % workload)
    try:
        txt = open(path).read()
    except OSError:
        return None
    vals = {}
    for line in txt.splitlines():
        if ":" in line and line.strip().startswith("- "):
            k, v = line.strip()[2:].split(":", 1)
            vals[k.strip()] = v.strip().strip("`")
    if vals.get("source_sha256") != rowpass_source_hash():
        return None
    if top_k > 0 and vals.get("top_k") != str(top_k):
        return None
    try:
        return float(vals["traffic_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def run_traffic(workload: str, args):
    """profiled_traffic for this run's filters: nucleus (top-p without top-k)
    and penalty rows run another row-pass variant, with no committed summary."""
    if args.rep_penalty != 1.0 or (args.top_k <= 0 and args.top_p < 1.0):
        return None
    return profiled_traffic(workload, args.top_k)


def algorithmic_bytes(wl, mp) -> dict:
    """Bytes the step must read once: every distinct mapped draft row and all
    m_b + 1 target rows of every request."""
    import numpy as np
    esz_d = wl.draft_logits.element_size()
    esz_t = wl.target_logits.element_size()
    rows_d = 0
    for b in range(wl.B):
        t0, t1 = int(wl.target_off[b]), int(wl.target_off[b + 1])
        rows_d += len(np.unique(mp[t0:t1]))
    d = rows_d * wl.draft_logits.shape[1] * esz_d
    t = (wl.n_target + wl.B) * wl.target_logits.shape[1] * esz_t
    return {"draft_rows": rows_d, "target_rows": wl.n_target + wl.B, "draft_bytes": d,
            "target_bytes": t, "total": d + t}


def default_steps(name: str) -> int:
    return {"b1_g4_v32k": 20000, "b64_g8_v152k": 20000, "b256_g16_v152k_bf16": 3000,
            "dtw_4096x64": 1000, "b1024_g8_v201k_bf16": 1000}.get(name, 1000)


def step_launches(args) -> int:
    """Kernels one tt_step launches: alignment, row pass and decision; with
    filters also the kept sets of top-k families, the nucleus kernel of
    top-p-only families and the transfer of q_hat before the decision."""
    pen = 1 if args.rep_penalty != 1.0 else 0  # the penalty's per-request sets
    if args.top_k > 0:
        return 5 + pen
    if args.top_p < 1.0:
        return 6  # the nucleus merge and the exact nucleus kernel
    return 3


def filters_config(args):
    """The sampling filters of the run for the config key (None without any)."""
    if args.top_k <= 0 and args.top_p >= 1.0 and args.rep_penalty == 1.0:
        return None
    f = {"top_k": args.top_k, "top_p": args.top_p}
    if args.rep_penalty != 1.0:
        f["rep_penalty"] = args.rep_penalty
        f["history"] = "64-1024 tokens per request and family"
    return f


def step_kwargs(args) -> dict:
    """The run's step parameters beyond the workload's own, for the oracle legs:
    the temperature override and the sampling filters of both families."""
    kw = {"top_k_draft": args.top_k, "top_k_target": args.top_k,
          "top_p_draft": args.top_p, "top_p_target": args.top_p}
    if args.rep_penalty != 1.0:
        kw["rep_penalty_draft"] = kw["rep_penalty_target"] = args.rep_penalty
    if args.temp is not None:
        kw["temp_draft"] = kw["temp_target"] = args.temp
    return kw


def oracle_sample_rate(wl, budget_s: float, step_kw=None, keep: bool = False):
    """Times the oracle (as it stands) over requests of the workload, cycling
    through them until the CPU budget is spent; returns positions/s, a note,
    the requests and seconds, and (keep=True) each request's first oracle
    result with its one-request workload."""
    import oracle
    oracle.build()
    order = list(range(wl.B))
    subs, outs = {}, {}
    done_req, positions, elapsed = 0, 0, 0.0
    while elapsed < budget_s:
        b = order[done_req % wl.B]
        if b not in subs:
            subs[b] = wl.subset([b])
        sw = subs[b]
        t = time.perf_counter()
        o = oracle.step(sw, request_base=b, **(step_kw or {}))
        elapsed += time.perf_counter() - t
        if keep and b not in outs:
            outs[b] = (sw, o)
        positions += int(sw.draft_off[-1])
        done_req += 1
    sample = ("%d requests of the %s batch (cycling from request 0), oracle single-threaded, "
              "fp64, %.1f s of CPU time" % (done_req, wl.spec.name, elapsed))
    if keep:
        return positions / elapsed, sample, done_req, elapsed, outs
    return positions / elapsed, sample, done_req, elapsed


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _oracle_job(job):
    """One worker process: the oracle, as it stands, over its list of requests
    (cycling) until `budget` seconds are spent (or once through when budget is
    0), with the step parameters `kw`; returns (positions, seconds, requests)."""
    subs, budget, kw = job
    import oracle
    oracle.build()
    positions, elapsed, done = 0, 0.0, 0
    i = 0
    while (budget > 0 and elapsed < budget) or (budget <= 0 and i < len(subs)):
        b, sw = subs[i % len(subs)]
        t = time.perf_counter()
        oracle.step(sw, request_base=b, **kw)
        elapsed += time.perf_counter() - t
        positions += int(sw.draft_off[-1])
        done += 1
        i += 1
    return positions, elapsed, done


def oracle_pool(n: int):
    """A pool of n oracle workers (spawned: never forked from a CUDA process)."""
    import multiprocessing
    return multiprocessing.get_context("spawn").Pool(n)


def oracle_all_cores_rate(wl, budget_s: float, per_worker: int = 2, step_kw=None):
    """The oracle on every host core: worker w cycles over its own `per_worker`
    requests of the batch for budget_s seconds; the rate is the sum of the
    workers' rates (each timed inside its process, without the pool's I/O)."""
    n = host_cores()
    jobs = []
    for w in range(n):
        idx = [(w * per_worker + i) % wl.B for i in range(per_worker)]
        jobs.append(([(b, wl.subset([b])) for b in idx], budget_s, step_kw or {}))
    with oracle_pool(n) as pool:
        res = pool.map(_oracle_job, jobs, chunksize=1)
    rate = sum(p / e for p, e, _ in res if e > 0)
    done = sum(d for _, _, d in res)
    sample = ("%d requests of the %s batch, %d per worker, one oracle process per host core "
              "(%d), fp64, %.1f s each" % (done, wl.spec.name, per_worker, n, budget_s))
    return rate, sample, n


# -------------------------------------------------------------- my arm

EXTRA_WORKLOADS = ("b64_g8_v152k", "b256_g16_v152k_bf16", "dtw_4096x64", "b1_g4_v32k")


def prepare_step(tt, W, name, args, rank, dev, stream):
    """The workload's inputs on the device, its step parameters, one untimed
    step with every output (mapped draft rows, acceptance, the parity sample),
    and a prepared call for the timed loop."""
    wl = W.make_workload(name, B=args.batch, seed=rank, device=str(dev))
    if args.rep_penalty != 1.0:
        wl = W.with_histories(wl, 64, 1024, seed=rank)
    inp = tt.device_inputs(wl, dev)
    prm = inp["params"]
    prm.request_base = request_base(rank, wl.B)
    if args.temp is not None:
        prm.temp_draft = prm.temp_target = args.temp
    prm.top_k_draft = prm.top_k_target = args.top_k
    prm.top_p_draft = prm.top_p_target = args.top_p
    prm.rep_penalty_draft = prm.rep_penalty_target = args.rep_penalty
    full = tt.tt_step(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                      inp["target_logits"], prm)
    import torch
    torch.cuda.synchronize(dev)
    assert int((full["status"] != 0).sum()) == 0, "a request failed"
    call = tt.StepCall(inp["batch"], inp["vd"], inp["vt"], inp["draft_logits"],
                       inp["target_logits"], prm,
                       out=tt.step_outputs(inp["batch"], dev, full=False), stream=stream)
    return wl, inp, prm, full, call


def time_steps(call, K, Wm, stream, dev, ws):
    """W untimed steps, then exactly K steps bracketed by a barrier and a device
    synchronise on both sides, timed with CUDA events on the launching stream.
    Stage events sit on at most one timed step in ten (events between the
    kernels break their dependent-launch overlap). Returns the time of the K
    steps (seconds, this rank), the host interval and the mean stage times."""
    import torch
    stride = max(10, math.ceil(K / 2000))
    sampled = list(range(0, K, stride))
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in sampled]
    for e4 in ev:
        for e in e4:
            e.record(stream)
    handles = [[e.cuda_event for e in e4] for e4 in ev]
    for _ in range(Wm):
        call()
    torch.cuda.synchronize(dev)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    barrier(ws)
    torch.cuda.synchronize(dev)
    h0 = time.perf_counter()
    t_start.record(stream)
    si = 0
    for i in range(K):
        if si < len(sampled) and sampled[si] == i:
            call(handles[si])
            si += 1
        else:
            call()
    t_end.record(stream)
    torch.cuda.synchronize(dev)
    h1 = time.perf_counter()
    barrier(ws)
    sec = t_start.elapsed_time(t_end) / 1e3
    stages = {"align": statistics.mean(e4[0].elapsed_time(e4[1]) for e4 in ev),
              "rowpass": statistics.mean(e4[1].elapsed_time(e4[2]) for e4 in ev),
              "decide": statistics.mean(e4[2].elapsed_time(e4[3]) for e4 in ev),
              "sampled_steps": len(sampled)}
    return sec, (h0, h1), stages


def extra_workload(tt, W, name, args, rank, ws, dev, stream, clocks, peak):
    """Another workload, timed in the same run as the headline one and with the
    same rules (its own K steps after W warm-up steps, inputs resident in HBM):
    the step time, the metric, the step's and the row pass's HBM rate, and the
    DTW alignment's pairs per second alone."""
    import numpy as np
    import torch
    wl, inp, prm, full, call = prepare_step(tt, W, name, args, rank, dev, stream)
    K = args.steps if args.steps is not None else min(default_steps(name), 2000)
    Wm = max(3, args.warmup)
    ab = algorithmic_bytes(wl, full["map"].cpu().numpy())
    sec, (h0, h1), st = time_steps(call, K, Wm, stream, dev, ws)
    sec_max = max_over_ranks(sec, ws, dev)
    align_alone_ms = run_align_alone(tt, wl, inp, prm, dev, stream)
    acc = full["accepted"].cpu().numpy()
    m = np.diff(wl.target_off)
    row_gbs = ab["total"] / (st["rowpass"] / 1e3) / 1e9
    r = {"workload": name, "batch_per_gpu": wl.B, "gamma": wl.spec.k,
         "dtype": "bf16" if wl.target_logits.element_size() == 2 else "f32", "steps": K,
         "ms_per_step": sec_max * 1e3 / K, "value": wl.n_draft * K * ws / sec_max,
         "unit": UNIT, "algorithmic_bytes": ab["total"],
         "hbm_gbs_step": ab["total"] / (sec / K) / 1e9,
         "step_frac_of_8tbs": ab["total"] / (sec / K) / 8e12,
         "rowpass_gbs": row_gbs, "rowpass_frac": row_gbs / peak,
         "rowpass_traffic": run_traffic(name, args),
         "stage_ms": st, "dtw_pairs_per_s": wl.B / (align_alone_ms / 1e3),
         "accept_rate": float(acc.sum() / max(1, m.sum())), "clocks": clocks.summary(h0, h1)}
    del wl, inp, full, call
    torch.cuda.empty_cache()
    return r


def cpu_baseline_leg(wl, full, args, step_kw):
    """The oracle, as it stands, on the host: one core over a bounded sample of
    the workload's requests (cycling from request 0), then one process per
    host core. The single-core sample's oracle outputs are also compared with
    the device step's outputs for the same requests (the untimed full step,
    launched as the timed ones), which gives the boundary-case counts the
    parity contract reports: accept decisions, drawn tokens and top-p cuts that
    differ within 1e-6 of their boundary, and any difference outside it."""
    from oracle.compare import compare_step
    rate, sample, nreq, el, outs = oracle_sample_rate(wl, args.cpu_seconds, step_kw,
                                                      keep=True)
    cpu = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample}
    g = {k: v.cpu().numpy() for k, v in full.items()}
    tot = {"requests_compared": 0, "accept_boundary": 0, "token_boundary": 0,
           "filter_boundary": 0, "mismatches": 0}
    first = []
    for b, (sw, o) in sorted(outs.items()):
        r = compare_step(g, o, sw.draft_off, sw.target_off, g_draft_off=wl.draft_off,
                         g_target_off=wl.target_off, req_index=[b])
        tot["requests_compared"] += 1
        for k in ("accept_boundary", "token_boundary", "filter_boundary"):
            tot[k] += r[k]
        tot["mismatches"] += len(r["mismatches"])
        first += r["mismatches"][:2]
    tot["first_mismatches"] = first[:4]
    tot["note"] = ("requests %s of the full-size step compared with the oracle: integers "
                   "exact, probabilities 1e-5 absolute and 1e-4 relative, a sampled result "
                   "excused only at the decision within 1e-6 of its boundary"
                   % ("0..%d" % (tot["requests_compared"] - 1)))
    rate, sample, n = oracle_all_cores_rate(wl, min(args.cpu_seconds, 8.0), step_kw=step_kw)
    cpu_all = {"value": rate, "unit": UNIT, "cores": n, "kind": "oracle", "sample": sample}
    return cpu, cpu_all, tot


def run_mine(args):
    import numpy as np
    import torch

    rank, ws, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist_init(ws, "nccl")
    import paper_2510_15545_gb300 as tt
    from paper_2510_15545_gb300 import workload as W
    tt.load(build_if_missing=(rank == 0 or ws == 1))
    barrier(ws)
    tt.load()

    name = args.workload
    K = args.steps if args.steps is not None else default_steps(name)
    Wm = max(3, args.warmup)
    stream = torch.cuda.current_stream(dev)
    wl, inp, prm, full, call = prepare_step(tt, W, name, args, rank, dev, stream)
    filtered = args.top_k > 0 or args.top_p < 1.0
    dl, tl = inp["draft_logits"], inp["target_logits"]
    mp = full["map"].cpu().numpy()
    acc = full["accepted"].cpu().numpy()
    ab = algorithmic_bytes(wl, mp)
    m = np.diff(wl.target_off)

    clocks = ClockSampler(local)
    time.sleep(0.3)
    sec, (h0, h1), st = time_steps(call, K, Wm, stream, dev, ws)
    sec_max = max_over_ranks(sec, ws, dev)
    clk = clocks.summary(h0, h1)
    align_ms, row_ms = st["align"], st["rowpass"]

    positions = wl.n_draft  # verified draft positions per step (batch x gamma)
    value = positions * K * ws / sec_max
    peak, peak_kind = measured_hbm_peak()
    achieved = ab["total"] / (row_ms / 1e3) / 1e9
    step_gbs = ab["total"] / (sec / K) / 1e9
    traffic = run_traffic(name, args)

    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(tt, wl, inp, prm, dev, stream, K, ws)

    align_alone_ms = run_align_alone(tt, wl, inp, prm, dev, stream)
    reenc = None if args.no_reencode else run_reencode(tt, wl, inp, prm, dev, stream, rank, ws)
    verify = None
    if not filtered and not prm.full_q:
        verify = run_verify_alone(tt, wl, inp, prm, full["q_hat"], dev, stream)
    cells = band_cells(wl, prm.window)
    sharded = None
    if args.shards > 0 and not filtered and not prm.full_q:
        sharded = run_sharded(tt, wl, inp, prm, full["q_hat"], dev, stream, args.shards)

    cpu = cpu_all = bnd = None
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        cpu, cpu_all, bnd = cpu_baseline_leg(wl, full, args, step_kwargs(args))

    extras = {}
    if not args.no_extra and args.batch is None:
        keep = dict(wl=wl, dl_shape=list(dl.shape), tl_shape=list(tl.shape),
                    in_bytes=dl.numel() * dl.element_size() + tl.numel() * tl.element_size())
        del inp, full, call, dl, tl
        torch.cuda.empty_cache()
        for x in EXTRA_WORKLOADS:
            if x != name:
                extras[x] = extra_workload(tt, W, x, args, rank, ws, dev, stream, clocks, peak)
        wl = keep["wl"]
        dl_shape, tl_shape, in_bytes = keep["dl_shape"], keep["tl_shape"], keep["in_bytes"]
    else:
        dl_shape, tl_shape = list(dl.shape), list(tl.shape)
        in_bytes = dl.numel() * dl.element_size() + tl.numel() * tl.element_size()
    time.sleep(0.2)
    clocks.stop()

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": K,
        "warmup": Wm, "ms_per_step": sec_max * 1e3 / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if wl.target_logits.element_size() == 2 else "f32",
        "data": "synthetic (seeded byte-string vocabularies, greedy re-encoding, Zipf logits)",
        "config": {"workload": name, "batch_per_gpu": wl.B, "gamma": wl.spec.k,
                   "V_d": wl.spec.V_d, "V_t": wl.spec.V_t,
                   "logits_cols": [int(dl_shape[1]), int(tl_shape[1])],
                   "target_tokens_per_gpu": wl.n_target, "window": prm.window,
                   "temperature": [prm.temp_draft, prm.temp_target],
                   "filters": filters_config(args),
                   "parallelism": "dp%d (independent requests per GPU)" % ws,
                   "l2": "inputs %.0f MB exceed the 129 MB L2; no flush between steps"
                         % (in_bytes / 1e6) if ab["total"] > L2_BYTES else "inputs fit in L2",
                   "accept_rate": float(acc.sum() / max(1, m.sum())),
                   "mean_accepted": float(acc.mean())},
        "hbm_gbs_step": step_gbs,
        "step_frac_of_8tbs": step_gbs / 8000.0,
        "dtw_pairs_per_s": wl.B / (align_alone_ms / 1e3),
        "dtw": {"ms_alone": align_alone_ms, "ms_in_step": align_ms,
                "pairs_per_s_in_step": wl.B / (align_ms / 1e3),
                "band_cells": cells, "band_cells_per_s": cells / (align_alone_ms / 1e3),
                "note": "dtw_pairs_per_s: tt_align alone (one warp per pair), 200 calls; in "
                        "the step the alignment takes one CTA per SM beside the row pass"},
        "stage_ms": st,
        "roofline": {"bound": "hbm", "kernel": "rowpass_kernel", "achieved": achieved,
                     "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                     "peak_kind": "%s copy bandwidth (hbm_gbs)" % peak_kind,
                     "traffic": traffic, "algorithmic_bytes": ab["total"],
                     "vs_nominal_8tbs": achieved / 8000.0},
        "gpu_launches": step_launches(args) * K,
        "clocks": clk,
    }
    if e2e is not None:
        line["e2e"] = e2e
    if reenc is not None:
        line["reencode"] = reenc
    if verify is not None:
        line["verify"] = verify
    if sharded is not None:
        line["sharded"] = sharded
    if cpu is not None:
        line["cpu_baseline"] = cpu
    if cpu_all is not None:
        line["cpu_baseline_all_cores"] = cpu_all
    if bnd is not None:
        line["boundary_cases"] = bnd
    if extras:
        line["workloads"] = extras
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def _time_calls(fn, stream, n, warm=3):
    import torch
    for _ in range(warm):
        fn()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    e0.record(stream)
    for _ in range(n):
        fn()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / n  # ms per call


def run_align_alone(tt, wl, inp, prm, dev, stream):
    """tt_align on its own (DTW and the map i*(j), nothing after it), timed with
    CUDA events over repeated calls outside the step's timed region. Alone it
    takes one warp per pair and as many CTAs as fit; inside tt_step the same
    kernel runs on one CTA per SM so that the row pass streams beside it."""
    call = tt.AlignCall(inp["batch"], inp["vd"], inp["vt"], prm, stream=stream)
    return _time_calls(call, stream, 200)


def band_cells(wl, window: int) -> int:
    """DTW cells inside the band over the whole batch: pairs (i, j), 1 <= i <= k,
    1 <= j <= m, with |i - j| <= max(w, |k - m|) (every cell when w < 0)."""
    import numpy as np
    k = np.diff(np.asarray(wl.draft_off, dtype=np.int64))
    m = np.diff(np.asarray(wl.target_off, dtype=np.int64))
    total = 0
    for kb, mb in zip(k.tolist(), m.tolist()):
        if window < 0:
            total += kb * mb
            continue
        W = max(window, abs(kb - mb))
        i = np.arange(1, kb + 1)
        total += int(np.maximum(0, np.minimum(mb, i + W) - np.maximum(1, i - W) + 1).sum())
    return total


def run_verify_alone(tt, wl, inp, prm, q_hat, dev, stream):
    """tt_verify on its own (target row pass and decision, with the step's
    q_hat), timed with CUDA events over repeated calls outside the step's timed
    region: the metric's positions over the verification alone."""
    batch, tl = inp["batch"], inp["target_logits"]
    ws_v = tt.binding.workspace(batch, 0, tl.shape[1], dev, prm)
    out = {}
    ms = _time_calls(lambda: out.update(tt.tt_verify(batch, q_hat, tl, prm, ws=ws_v, out=out,
                                                     stream=stream)), stream, 50)
    tbytes = (wl.n_target + wl.B) * tl.shape[1] * tl.element_size()
    return {"ms_per_call": ms, "positions_per_s": wl.n_draft / (ms / 1e3),
            "target_bytes": tbytes, "target_gbs": tbytes / (ms / 1e3) / 1e9,
            "note": "tt_verify alone on the step's q_hat, 50 calls"}


def run_sharded(tt, wl, inp, prm, q_hat, dev, stream, S):
    """The verification of the batch's target rows split by columns into S
    near-equal slices held in separate arrays (tt_verify_sharded: per-shard row
    passes, the gathered records, the merged decision), against tt_verify on the
    unsplit rows with the same q_hat; each timed alone with CUDA events over
    repeated calls, outside the step's timed region. Also reports how many
    requests the two agree on and the bytes an all-gather of the records moves."""
    import torch
    tl = inp["target_logits"]
    V = tl.shape[1]
    per16 = 16 // tl.element_size()
    cuts = [round(V * k / S) for k in range(S + 1)]
    shards = []
    for a, b in zip(cuts, cuts[1:]):
        buf = torch.empty((tl.shape[0], (b - a + per16 - 1) // per16 * per16), dtype=tl.dtype,
                          device=dev)
        buf[:, :b - a] = tl[:, a:b]
        shards.append(buf[:, :b - a])
    batch = inp["batch"]
    ws_v = tt.binding.workspace(batch, 0, V, dev, prm)
    ws_s = tt.binding.sharded_workspace(batch, shards, dev)
    out_v, out_s = {}, {}
    unsplit = lambda: out_v.update(tt.tt_verify(batch, q_hat, tl, prm, ws=ws_v, out=out_v,
                                                 stream=stream))
    split = lambda: out_s.update(tt.tt_verify_sharded(batch, q_hat, shards, prm, ws=ws_s,
                                                       out=out_s, stream=stream))
    n = 50
    t_unsplit = _time_calls(unsplit, stream, n)
    t_split = _time_calls(split, stream, n)
    rows = batch.n_target + batch.B
    agree_a = int((out_v["accepted"] == out_s["accepted"]).sum())
    agree_t = int((out_v["next_token"] == out_s["next_token"]).sum())
    return {"shards": S, "verify_ms_unsplit": t_unsplit, "verify_ms_sharded": t_split,
            "exchange_bytes": 16 * S * rows, "requests": batch.B,
            "agree_accepted": agree_a, "agree_next_token": agree_t}


def run_reencode(tt, wl, inp, prm, dev, stream, rank, ws):
    """The re-encoding of the batch's draft strings into target tokens on the
    device (tt_encode), its Lemma-1 check (tt_consistency) and the delta-pos
    histogram of the alignment paths (tt_dpos_hist), each timed alone with CUDA
    events over repeated calls; and, on rank 0, the oracle's re-encoding of the
    same batch on one host core. Outside the step's timed region: re-encoding
    precedes the target model's forward, it is not part of a verification step."""
    import time

    import numpy as np
    import torch
    index = tt.vocab_index(wl.vt.blob, wl.vt.off, dev)
    d_off, d_ids = inp["batch"].draft_off, inp["batch"].draft_ids
    max_m = 512
    ws_enc = torch.empty(max(tt.tt_encode_workspace_bytes(wl.B, max_m), 256), dtype=torch.uint8,
                         device=dev)
    out = {"target_off": torch.empty(wl.B + 1, dtype=torch.int32, device=dev),
           "target_ids": torch.empty(wl.B * max_m, dtype=torch.int32, device=dev),
           "status": torch.empty(wl.B, dtype=torch.int32, device=dev)}
    enc = lambda: tt.tt_encode(d_off, d_ids, inp["vd"], inp["vt"], index, max_m, out=out,
                               ws=ws_enc, stream=stream)
    enc_ms = _time_calls(enc, stream, 200)
    n_out = int(out["target_off"][-1])
    ok = int((out["status"] == 0).sum())
    cons_status = torch.empty(wl.B, dtype=torch.int32, device=dev)
    cons_ms = _time_calls(lambda: tt.tt_consistency(inp["batch"], inp["vd"], inp["vt"],
                                                    status=cons_status, stream=stream), stream, 200)
    prm0 = tt.Params(window=-1, seed=prm.seed)
    al = tt.tt_align(inp["batch"], inp["vd"], inp["vt"], prm0)
    hist = torch.zeros(64, dtype=torch.int64, device=dev)
    dpos_ms = _time_calls(lambda: tt.tt_dpos_hist(inp["batch"], al["path"], al["path_len"],
                                                  al["map"], 0, 64, hist=hist, stream=stream),
                          stream, 200)
    h = tt.tt_dpos_hist(inp["batch"], al["path"], al["path_len"], al["map"], 0, 64).cpu().numpy()
    cdf = np.cumsum(h) / max(1, h.sum())
    r = {"draft_tokens": wl.n_draft, "target_tokens": n_out, "requests_ok": ok,
         "encode_ms_per_batch": enc_ms,
         "encode_draft_tokens_per_s": wl.n_draft / (enc_ms / 1e3),
         "consistency_ms_per_batch": cons_ms, "dpos_hist_ms_per_batch": dpos_ms,
         "dpos_cdf_0.9_at": int(np.searchsorted(cdf, 0.9)),
         "bound": "latency (dependent L2 probes of the prefix index; a few KB per request)"}
    if rank == 0 and ws == 1:
        import oracle
        oracle.build()
        t0 = time.process_time()
        oracle.encode(wl.draft_off, wl.draft_ids, wl.vd.blob, wl.vd.off, wl.vt.blob, wl.vt.off,
                      max_m)
        cpu_s = time.process_time() - t0
        r["cpu_oracle_encode_ms_per_batch"] = cpu_s * 1e3
        r["cpu_oracle_note"] = ("the oracle re-encodes the whole batch on one host core (its "
                                "vocabulary sort included, as in one call)")
    return r


def run_e2e(tt, wl, inp, prm, dev, stream, K, ws):
    """The same metric through the public API with the step's inputs in pinned
    host memory: every step copies ids, offsets and logits host -> device,
    runs tt_step and reads the results back. Two sets of device inputs let the
    copy of step i + 1 (on its own stream) run while step i computes."""
    import torch

    def dev_list(d):
        b = d["batch"]
        t = [b.draft_off, b.draft_ids, b.target_off, b.target_ids, b.draft_cols, b.target_cols,
             d["draft_logits"], d["target_logits"]]
        return [x for x in t if x is not None]

    sets = [inp, tt.device_inputs(wl, dev)]
    host = [t.cpu().pin_memory() for t in dev_list(inp)]
    calls, outs = [], []
    for d in sets:
        out = tt.step_outputs(d["batch"], dev, full=False)
        outs.append(out)
        calls.append(tt.StepCall(d["batch"], d["vd"], d["vt"], d["draft_logits"],
                                 d["target_logits"], prm, out=out, stream=stream))
    keys = ("accepted", "next_token", "status")
    res_host = [[torch.empty_like(o[k], device="cpu").pin_memory() for k in keys] for o in outs]
    h2d = sum(t.numel() * t.element_size() for t in host)
    d2h = sum(t.numel() * t.element_size() for t in res_host[0])
    copy_stream = torch.cuda.Stream(dev)
    copied = [torch.cuda.Event() for _ in sets]
    done = [torch.cuda.Event() for _ in sets]
    for e in done:
        e.record(stream)

    def steps(n):
        for i in range(n):
            s = i % 2
            copy_stream.wait_event(done[s])  # step i - 2 has finished with set s
            with torch.cuda.stream(copy_stream):
                for d, h in zip(dev_list(sets[s]), host):
                    d.copy_(h, non_blocking=True)
            copied[s].record(copy_stream)
            stream.wait_event(copied[s])
            calls[s]()
            for h, k in zip(res_host[s], keys):
                h.copy_(outs[s][k], non_blocking=True)
            done[s].record(stream)
        stream.synchronize()
        copy_stream.synchronize()

    steps(4)
    t0 = time.perf_counter()
    steps(2)
    est = (time.perf_counter() - t0) / 2
    n = max(3, min(K, int(math.ceil(3.0 / max(est, 1e-6)))))
    barrier(ws)
    t0 = time.perf_counter()
    steps(n)
    sec = time.perf_counter() - t0
    sec = max_over_ranks(sec, ws, dev)
    return {"value": wl.n_draft * n * ws / sec, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": n, "ms_per_step": sec * 1e3 / n,
            "api": "pinned host tensors -> copy_(non_blocking, copy stream) -> tt_step -> "
                   "copy_ back; two input sets, the copy of step i + 1 overlapping step i"}


# ---------------------------------------------------------- reference arm

def run_reference(args):
    """The CPU oracle as it stands, on the host cores, on the same workload and
    metric: each step is a bounded sample of the batch's requests."""
    rank, ws, local = dist_env()
    if rank != 0:
        return
    from paper_2510_15545_gb300 import workload as W
    import oracle
    oracle.build()
    name = args.workload
    K = args.steps if args.steps is not None else 5
    Wm = max(3, args.warmup)
    import torch
    # the same draws as the GPU arm's (its generator runs on the device); the
    # oracle reads each request's rows copied to the host
    gen_dev = "cuda" if torch.cuda.is_available() else "cpu"
    wl = W.make_workload(name, B=args.batch, seed=0, device=gen_dev)
    if args.rep_penalty != 1.0:
        wl = W.with_histories(wl, 64, 1024, seed=0)
    per_worker = {"b1_g4_v32k": 1, "b64_g8_v152k": 2, "b256_g16_v152k_bf16": 1,
                  "dtw_4096x64": 8, "b1024_g8_v201k_bf16": 1}.get(name, 1)
    n = host_cores()
    kw = step_kwargs(args)
    spec = wl.spec
    temps = [kw.get("temp_draft", spec.temp_draft), kw.get("temp_target", spec.temp_target)]
    # step s: worker w takes requests ((s * n + w) * per_worker + i) mod B; a
    # step's time is the slowest worker's oracle time (measured in the worker)
    def step_jobs(s):
        jobs = []
        for w in range(n):
            idx = [((s * n + w) * per_worker + i) % wl.B for i in range(per_worker)]
            jobs.append(([(b, wl.subset([b])) for b in idx], 0.0, kw))
        return jobs
    sec, pos = 0.0, 0
    with oracle_pool(n) as pool:
        for s in range(Wm):
            pool.map(_oracle_job, step_jobs(s), chunksize=1)
        for s in range(Wm, Wm + K):
            res = pool.map(_oracle_job, step_jobs(s), chunksize=1)
            sec += max(e for _, e, _ in res)
            pos += sum(p for p, _, _ in res)
    value = pos / sec
    per_step = n * per_worker
    sample = ("%d requests of the %s batch per step, %d per oracle process, one process per "
              "host core (%d), fp64; a step lasts as long as its slowest process; inputs "
              "drawn on %s" % (per_step, name, per_worker, n, gen_dev))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": ws, "steps": K, "warmup": Wm, "ms_per_step": sec * 1e3 / K,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": name, "batch_per_gpu": wl.B, "gamma": spec.k,
                       "V_d": spec.V_d, "V_t": spec.V_t,
                       "logits_cols": [int(wl.draft_logits.shape[1]),
                                       int(wl.target_logits.shape[1])],
                       "target_tokens_per_gpu": wl.n_target, "window": spec.window,
                       "temperature": temps,
                       "filters": filters_config(args),
                       "parallelism": "oracle processes on the host cores",
                       "requests_per_step": per_step},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": n, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_mine(args)


if __name__ == "__main__":
    main()
