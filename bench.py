"""Benchmark of the gs-SGD compression step on GB300.

One step = the whole hot path for P simulated workers on one GPU: accumulate + Count
Sketch insert (fused), tree merge, median query + top-k, gather-and-zero.  The metric is
gradient coordinates per second, P * d * steps / time.  The headline workload is the
ResNet-50-sized one (d = 25,557,032, P = 8, r = 5, c = 2^18, k = 25,600) unless --config
names another; `per_config` in the same JSON line times every workload of the suite.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

Under torchrun (N > 1) every rank runs an independent replica of the workload on its own
GPU (weak scaling, no collective on the data path); rank 0 prints one JSON line.
--impl reference times the CPU oracle (the reference arm of this comparison) on bounded
samples of the same workload.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads  # noqa: E402

METRIC = "gradient coords/s through accumulate+sketch+merge+top-k at P=8; % HBM roofline"
UNIT = "coords/s"
DEFAULT_CONFIG = "resnet50"
CSRC = os.path.join(ROOT, "paper_2108_06004_gb300", "csrc")
TRAFFIC_JSON = os.path.join(ROOT, "profiles", "traffic.json")
CPU_SAMPLE_D = 1 << 22   # coordinates per worker in one bounded oracle step (CPU baseline)
REF_BUDGET_S = 120.0     # oracle seconds for a whole --impl reference run
ORACLE_S_PER_COORD = 1.7e-7  # oracle seconds per worker-coordinate (sizes the reference samples)
L2_BYTES = 126 << 20     # GB300 L2; inputs below twice this are flushed between timed steps
PER_CONFIG_STEPS = {"tiny-2^20": 300, "resnet18": 300, "resnet50": 100, "vgg16": 5, "bert-large": 3}
PRUNE_MIN_DIM = 1 << 22  # the library skips query rows from this dimension on
SAMPLE_PERIOD = 256      # ... with a prune-key sample of the first four of every 256 coordinates
CLASS_BYTES = 192 << 10  # ... and classifies the first r/2 + 1 rows in shared memory when they fit


def query_classifies(r: int, c: int) -> bool:
    """Whether a pruning query of r rows and c columns runs the shared-memory classification
    (one more kernel, which writes the cell classes)."""
    return 3 <= r <= 16 and c >= 64 and (c & (c - 1)) == 0 and (r // 2 + 1) * c // 4 <= CLASS_BYTES

VARIANTS = {
    "error_feedback": "S1-S6: per-worker momentum and error vectors, exact second round",
    "train": "S1-S7: as error_feedback, with the weight update fused into the second round",
    "heavymix": "S1-S6 with the HEAVYMIX selection in place of the top-k",
    "sketched_state": "momentum and error kept as r x c sketches; no per-worker state vectors",
}
HEAVYMIX_FILL_SEED = 0x5EED5EED
LR = 0.01


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default=DEFAULT_CONFIG, choices=sorted(workloads.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--variant", default="error_feedback", choices=list(VARIANTS),
                    help="which form of the step to time (the default is the headline path)")
    ap.add_argument("--eager", action="store_true",
                    help="one library call per kernel instead of a captured plan per step")
    ap.add_argument("--group-width", type=int, default=0,
                    help="workers interleaved per sketch table (0: the library's choice)")
    ap.add_argument("--insert", default="direct", choices=["direct", "staged"],
                    help="staged: the shared-memory-staged insert (gs_accumulate_insert_staged; eager, and only "
                         "where a table row fits a shared-memory tile)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-config", action="store_true", help="time only the headline workload")
    ap.add_argument("--profile-steps", action="store_true",
                    help="short run for a profiler: no e2e, no CPU baseline, no clocks, no probes, no per-config")
    ap.add_argument("--d", type=int, default=0,
                    help="profiling a small case: the workload's first D coordinates (its leading blocks, the "
                         "last one cut), same P, r, c and k scaled with D; implies --profile-steps")
    return ap.parse_args(argv)


def shrink(w, d: int):
    """The workload restricted to its first d coordinates (blocks cut at d; k scaled with d)."""
    import dataclasses
    blocks, tot = [], 0
    for b in w.blocks:
        if tot >= d:
            break
        blocks.append(min(b, d - tot))
        tot += blocks[-1]
    return dataclasses.replace(w, d=d, k=max(1, round(w.k * d / w.d)), block_sizes=tuple(blocks),
                               name=f"{w.name}@d={d}")


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}, "fallback"


# ---- clocks ------------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi samples every 50 ms of the GPU (selected by UUID); stop() keeps the samples
    whose own timestamps fall in the timed window (or, for a window shorter than the sampling
    period, the samples nearest to it)."""
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu = gpu_id
        self.proc = None
        self.t0 = self.t1 = None

    def start(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-i", self.gpu,
               "-lms", "50"]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.5)

    def mark_begin(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def stop(self):
        import datetime
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        time.sleep(0.2)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        inside = [x for x in rows if self.t0 <= x[0] <= self.t1]
        if not inside and rows:
            mid = 0.5 * (self.t0 + self.t1)
            inside = sorted(rows, key=lambda x: abs(x[0] - mid))[:2]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        reasons = sorted({n for x in inside for n, f in zip(self.NAMES, x[3]) if f.lower().startswith("active")})
        return {"sm_mhz": statistics.median(x[1] for x in inside), "sm_max_mhz": max(x[2] for x in inside),
                "reasons": reasons, "samples": len(inside),
                "window_s": round(self.t1 - self.t0, 3)}


# ---- ncu traffic ------------------------------------------------------------------------

def source_sha16(name: str) -> str:
    return hashlib.sha256(open(os.path.join(CSRC, name), "rb").read()).hexdigest()[:16]


def measured_traffic(kernel: str, workload: str):
    """DRAM bytes (read + write) per launch of `kernel` on `workload` from profiles/traffic.json
    (written from one ncu capture, scaled to a full launch where the capture was smaller), if
    it was taken on the current source of the kernel's file; else None."""
    try:
        with open(TRAFFIC_JSON) as f:
            entry = json.load(f)["kernels"][kernel][workload]
    except (OSError, KeyError, ValueError):
        return None
    if entry.get("source_sha16") != source_sha16(entry["source"]):
        return None
    return entry.get("dram_bytes_per_full_launch")


# ---- ranks --------------------------------------------------------------------------------

def dist_max(x: float, device=None) -> float:
    """The maximum of x over all ranks (x itself without an initialised process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_workers(rank: int, P: int) -> list:
    """Worker ids whose gradients rank `rank` draws: independent replicas per rank."""
    return [rank * P + p for p in range(P)]


def whole_job_rate(world: int, P: int, d: int, steps: int, max_seconds: float) -> float:
    """Worker-coordinates of all ranks per second of the slowest rank."""
    return world * P * d * steps / max_seconds


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def gpu_uuid(dev) -> str:
    import torch
    u = str(torch.cuda.get_device_properties(dev).uuid)
    return u if u.startswith("GPU-") else "GPU-" + u


# ---- one workload ---------------------------------------------------------------------------

def _event_pair(record):
    import torch
    if not record:
        return None
    return torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)


class Runner:
    """Everything one workload's timed steps need: state, sketches, workspace, gradients and,
    unless eager, one plan (CUDA graph) per gradient buffer set.

    Workloads whose P workers are all resident draw a pool of fresh gradient sets (one per step
    of the workload, as many as fit 24 GB), cycled over the timed steps.  A workload with a
    worker batch (BERT-large: 32 workers, 8 resident) streams: every step, for each batch, the
    batch's fresh gradients are drawn on the device into one shared buffer set (timed with
    their own events, outside the insert's) and then inserted; such steps run eagerly."""

    def __init__(self, gs, w, variant, eager, rank, dev, stream, steps_needed, want_host_pool, staged=False,
                 group_width=0):
        import torch
        self.gs, self.w, self.variant, self.dev, self.stream = gs, w, variant, dev, stream
        self.staged = staged
        if staged:
            eager = True
        self.rank = rank
        P, d, r, c, k = w.P, w.d, w.r, w.c, w.k
        self.streamed = bool(w.worker_batch) and w.worker_batch < P
        self.batch = w.worker_batch if self.streamed else P
        self.host_pool, self.dev_pool = [], []
        if self.streamed:
            self.gbuf = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(self.batch)]
            self.nsteps_pool = 1
        else:
            step_bytes = P * d * 4
            self.nsteps_pool = max(1, min(w.steps, steps_needed, (24 << 30) // step_bytes))
            host_gen = step_bytes <= (1 << 30)
            for t in range(self.nsteps_pool):
                if host_gen:
                    gl = workloads.make_gradients(w, t, replica_workers(rank, P))
                    hp = [torch.from_numpy(g).pin_memory() for g in gl]
                    if want_host_pool:
                        self.host_pool.append(hp)
                    self.dev_pool.append([g.to(dev, non_blocking=True) for g in hp])
                else:
                    self.dev_pool.append([workloads.make_gradient_torch(w, t, q, torch.empty(d, device=dev))
                                          for q in replica_workers(rank, P)])
            if want_host_pool and not host_gen:
                self.host_pool = [[g.cpu().pin_memory() for g in self.dev_pool[0]]]
        self.us = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
        self.es = [torch.zeros(d, dtype=torch.float32, device=dev) for _ in range(P)]
        gs = self.gs
        self.sk = gs.gs_sketch_create(r, c, 20210813, P, group_width)
        info = gs.gs_sketch_info(self.sk)
        self.W, self.rpp = info["group_width"], info["rows_per_pass"]
        self.groups = (P + self.W - 1) // self.W
        self.passes = -(-r // self.rpp)
        ws_bytes = gs.gs_step_workspace_size(d, k)
        if variant == "heavymix":
            ws_bytes = max(ws_bytes, gs.gs_query_heavymix_workspace_size(d, k))
        self.ws = torch.empty(ws_bytes, dtype=torch.uint8, device=dev)
        self.qws_bytes = gs.gs_query_topk_workspace_size(d, k)
        self.l2sq = torch.empty(1, dtype=torch.float64, device=dev)
        self.weights = torch.zeros(d, dtype=torch.float32, device=dev) if variant in ("train", "sketched_state") \
            else None
        self.sk_u = self.sk_e = None
        if variant == "sketched_state":
            self.sk_u = gs.gs_sketch_create(r, c, 20210813, 1, 0)
            self.sk_e = gs.gs_sketch_create(r, c, 20210813, 1, 0)
            gs.gs_sketch_zero(self.sk_u)
            gs.gs_sketch_zero(self.sk_e)
        self.idx = torch.empty(k, dtype=torch.int64, device=dev)
        self.vals = torch.empty(k, dtype=torch.float32, device=dev)
        self.use_plan = (not eager or variant == "sketched_state") and not self.streamed
        self.plans = []
        flags = gs.GS_PLAN_TIME_INSERT | gs.GS_PLAN_TIME_QUERY
        if self.use_plan:
            for grads in self.dev_pool:
                if variant == "sketched_state":
                    self.plans.append(gs.gs_sketched_state_plan_create(
                        self.sk, self.sk_u, self.sk_e, grads, d, w.rho, k, self.idx, self.vals, self.weights, LR,
                        self.ws, flags=flags))
                elif variant == "heavymix":
                    self.plans.append(gs.gs_heavymix_step_plan_create(
                        self.sk, self.us, self.es, grads, d, w.rho, k, HEAVYMIX_FILL_SEED, self.idx, self.vals,
                        self.l2sq, self.ws, flags=flags))
                else:
                    self.plans.append(gs.gs_step_plan_create(self.sk, self.us, self.es, grads, d, w.rho, k, self.idx,
                                                             self.vals, None, self.weights, LR, self.ws, flags=flags))
        self.ev = {"insert": [], "query": [], "gen": []}   # eager: per step, a list of (begin, end) pairs

    def step(self, t, record):
        gs, w, s = self.gs, self.w, self.stream
        d, k, rho = w.d, w.k, w.rho
        if self.use_plan:
            gs.gs_plan_launch(self.plans[t % self.nsteps_pool], s)
            return
        if self.variant == "sketched_state":
            raise RuntimeError("the sketched state always runs as a plan")
        gs.gs_sketch_zero(self.sk, s)
        if self.streamed:
            ins_pairs, gen_pairs = [], []
            for b0 in range(0, w.P, self.batch):
                gen = _event_pair(record)
                if gen:
                    gen[0].record(s)
                for q in range(self.batch):
                    workloads.make_gradient_torch(w, t, self.rank * w.P + b0 + q, self.gbuf[q])
                if gen:
                    gen[1].record(s)
                    gen_pairs.append(gen)
                ins = _event_pair(record)
                if ins:
                    ins[0].record(s)
                gs.gs_accumulate_insert(self.sk, b0, self.us[b0:b0 + self.batch], self.es[b0:b0 + self.batch],
                                        self.gbuf, d, rho, s)
                if ins:
                    ins[1].record(s)
                    ins_pairs.append(ins)
            if record:
                self.ev["insert"].append(ins_pairs)
                self.ev["gen"].append(gen_pairs)
        else:
            ins = _event_pair(record)
            if ins:
                ins[0].record(s)
            insert = gs.gs_accumulate_insert_staged if self.staged else gs.gs_accumulate_insert
            insert(self.sk, 0, self.us, self.es, self.dev_pool[t % self.nsteps_pool], d, rho, s)
            if ins:
                ins[1].record(s)
                self.ev["insert"].append([ins])
        gs.gs_sketch_merge_tree(self.sk, w.P, s)
        q = _event_pair(record)
        if q:
            q[0].record(s)
        if self.variant == "heavymix":
            gs.gs_query_heavymix(self.sk, d, k, HEAVYMIX_FILL_SEED, self.idx, None, self.l2sq, self.ws, None, s)
        else:
            gs.gs_query_topk(self.sk, d, k, self.idx, None, self.ws, self.qws_bytes, s)
        if q:
            q[1].record(s)
            self.ev["query"].append([q])
        if self.variant == "train":
            gs.gs_gather_zero_update(self.us, self.es, d, self.idx, k, self.vals, self.weights, LR, s)
        else:
            gs.gs_gather_and_zero(self.us, self.es, d, self.idx, k, self.vals, s)

    def phase_times(self, n_timed_by_plan):
        """Mean ms of the insert phase, the median query (plans) and the selection (plans), or
        of the whole query + selection (eager), and of gradient generation (streamed)."""
        def mean(x):
            return sum(x) / len(x) if x else None
        if self.use_plan:
            ins, qry, sel = [], [], []
            for i, plan in enumerate(self.plans):
                n = n_timed_by_plan[i]
                if n:
                    ins += self.gs.gs_plan_insert_times(plan, n)
                    a, b = self.gs.gs_plan_query_times(plan, n)
                    qry += a
                    sel += b
            return {"insert": mean(ins), "query": mean(qry), "select": mean(sel), "query_select": None, "gen": None,
                    "n": len(ins)}
        def per_step(phase):   # each step's pairs summed (a streamed step has one per batch)
            return [sum(a.elapsed_time(b) for a, b in pairs) for pairs in self.ev[phase]]
        ins = per_step("insert")
        return {"insert": mean(ins), "query": None, "select": None, "query_select": mean(per_step("query")),
                "gen": mean(per_step("gen")), "n": len(ins)}

    def query_rows(self):
        """(fraction of coordinates that stopped early, rows examined per coordinate, table
        cells read per coordinate) in the last query: a coordinate that stopped after examining
        n rows, g of whose cells it read from the table, leaves -((32 g + n) * 2^-149) as its
        estimate; every other coordinate read all r cells."""
        import torch
        d, r = self.w.d, self.w.r
        bits = self.ws[: 4 * d].view(torch.int32)
        marked = (bits > -2**31) & (bits < -2**31 + 1024)
        n_marked = int(marked.sum().item())
        low = bits[marked].to(torch.int64) + 2**31
        examined = int((low & 31).sum().item())
        gathered = int((low >> 5).sum().item())
        return n_marked / d, (examined + (d - n_marked) * r) / d, (gathered + (d - n_marked) * r) / d

    def close(self):
        for plan in self.plans:
            self.gs.gs_plan_destroy(plan)
        self.plans = []
        for sk in (self.sk, self.sk_u, self.sk_e):
            if sk:
                self.gs.gs_sketch_destroy(sk)
        self.sk = self.sk_u = self.sk_e = None


def launches_per_step(run: Runner, variant: str) -> int:
    """Kernels of the library launched per step: insert (one per group and row pass, and per
    worker batch), merge, the query and selection, the gather (sketched state: its own)."""
    w = run.w
    prunes = variant != "heavymix" and w.d >= PRUNE_MIN_DIM and w.r >= 3 and (w.c & (w.c - 1)) == 0
    inserts = run.groups * run.passes
    if variant == "heavymix":
        query = 3 + 6                                 # sumsq, theta, query (with the keys) + selection
    else:
        # query + selection (+ sample and repair check, + the cell classes)
        query = 1 + 6 + (2 + int(query_classifies(w.r, w.c)) if prunes else 0)
    tail = 6 if variant == "sketched_state" else 1
    return inserts + 1 + query + tail


def time_steps(run: Runner, steps: int, warmup: int, world: int, dev, sampler=None, flush=None):
    """Run warm-up steps (every plan at least once), then time `steps` steps.  Without `flush`
    the timed region is bracketed by events on the stream; with it (inputs that fit in L2), a
    buffer larger than L2 is written before every timed step, outside that step's events."""
    import torch
    s = run.stream
    n_warm = max(warmup, len(run.plans))
    for t in range(n_warm):
        run.step(t, False)
    torch.cuda.synchronize()
    for k in run.ev:
        run.ev[k].clear()
    barrier(world)
    torch.cuda.synchronize()
    if sampler:
        sampler.mark_begin()
    if flush is None:
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(s)
        for t in range(steps):
            run.step(warmup + t, True)
        end.record(s)
        torch.cuda.synchronize()
        elapsed = start.elapsed_time(end)
    else:
        pairs = []
        for t in range(steps):
            flush.add_(1)
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(s)
            run.step(warmup + t, True)
            b.record(s)
            pairs.append((a, b))
        torch.cuda.synchronize()
        elapsed = sum(a.elapsed_time(b) for a, b in pairs)
    barrier(world)
    if sampler:
        sampler.mark_end()
    elapsed = dist_max(elapsed, dev)
    n_by_plan = [sum(1 for t in range(steps) if (warmup + t) % run.nsteps_pool == i) for i in range(len(run.plans))]
    return elapsed, n_warm, n_by_plan


def rooflines(run: Runner, variant: str, ph: dict, peaks, peak_kind, probes: dict, pruned: float,
              rows_read: float, cells_read: float):
    """The insert-phase roofline (HBM, with the measured request ceiling as co-bound) and the
    median query's (L1->L2 requests against the measured gather ceiling; HBM bytes alongside)."""
    w = run.w
    P, d, r = w.P, w.d, w.r
    per_wc = 4.0 if variant == "sketched_state" else 20.0
    moved_wc = per_wc + 4.0 * (run.passes - 1)   # every pass after the first re-reads e (or g)
    phase_s = ph["insert"] / 1e3
    phase_bytes = per_wc * P * d
    k1_gbs = phase_bytes / phase_s / 1e9
    cells = d * r * run.groups
    nl = run.groups * run.passes
    k1 = {
        "kernel": ("k_accumulate + k_insert_staged (S1, then S2 staged in shared memory" if run.staged else
                   "k_accumulate_insert_coop (insert only" if variant == "sketched_state" else
                   "k_accumulate_insert_coop (fused S1+S2") + f", W={run.W}), the insert phase of a step: "
                  f"{run.groups} group(s) x {run.passes} row pass(es)",
        "row_passes": run.passes, "groups": run.groups, "launches_per_phase": nl,
        "algorithmic_bytes_per_worker_coord": per_wc, "moved_bytes_per_worker_coord": moved_wc,
        "bound": "hbm", "achieved": round(k1_gbs, 1), "peak": peaks["hbm_gbs"], "unit": "GB/s",
        "frac": round(k1_gbs / peaks["hbm_gbs"], 4), "peak_source": peak_kind,
        "frac_of_nominal_8000_GBps": round(k1_gbs / 8000.0, 4),
        "traffic": (measured_traffic("k_accumulate_insert_coop", w.name)
                    if variant == "error_feedback" and nl == 1 else None),
        "algorithmic_bytes_per_launch": phase_bytes / nl if nl == 1 else None,
        "algorithmic_bytes_per_phase": phase_bytes,
        "avg_launch_ms": round(ph["insert"] / nl, 4),
        "avg_phase_ms": round(ph["insert"], 4),
        "timed_phases": ph["n"],
        "timing": "event-record nodes inside the step's CUDA graph" if run.use_plan else "CUDA events around the call",
    }
    # the probe stands for the fused accumulate + insert; the sketched state inserts raw gradients
    ceil_ms = probes.get("insert_ms") if variant != "sketched_state" else None
    k1["co_bound"] = {
        "kind": "SM->L2 requests: one cell reduction per (coordinate, row, group) plus the u, e stores and the loads",
        "probe": "gs_insert_request_ceiling: the same kernels, grids, buckets and reductions with every vector access "
                 "folded into an L2-resident window (no HBM traffic)",
        "cell_updates_per_phase": cells,
        "achieved_G_cells_per_s": round(cells / phase_s / 1e9, 1),
        "peak_ms": None if ceil_ms is None else round(ceil_ms, 4),
        "peak": None if ceil_ms is None else round(phase_bytes / (ceil_ms / 1e3) / 1e9, 1),
        "unit": "GB/s of algorithmic bytes",
        "frac": None if ceil_ms is None else round(ceil_ms / ph["insert"], 4),
        "peak_frac_of_hbm": None if ceil_ms is None else round(phase_bytes / (ceil_ms / 1e3) / 1e9 / peaks["hbm_gbs"], 4),
    }
    q = None
    q_ms = ph["query"]
    with_selection = q_ms is None and ph["query_select"] is not None   # eager: one pair of events per call
    if with_selection:
        q_ms = ph["query_select"]
    if q_ms is not None and variant != "heavymix":
        prunes = d >= PRUNE_MIN_DIM and r >= 3 and (w.c & (w.c - 1)) == 0
        nq = (d + 3) // 4
        n_s = 4 * ((nq + SAMPLE_PERIOD // 4 - 1) // (SAMPLE_PERIOD // 4)) if prunes else 0
        requests = d * cells_read + n_s * r
        g_ms = probes.get("query_ms")
        ach = requests / (q_ms / 1e3) / 1e9
        q = {
            "kernel": ((f"k_qsample + k_pbits + k_query_bits<{r}> + k_repair (median query, S4)"
                        if query_classifies(r, w.c) else f"k_qsample + k_query<{r}> + k_repair (median query, S4)")
                       if prunes else f"k_query<{r}> (S4)") +
                      (" and the S5 selection: eager, timed around the gs_query_topk call" if with_selection else ""),
            "bound": ("integer ALU pipe: the Mersenne hash of every row examined (the first rows' cells are "
                      "classified in shared memory, so few are read)" if prunes and query_classifies(r, w.c) else
                      "L1->L2 requests (scattered 4-byte reads of the merged table)"),
            "avg_ms": round(q_ms, 4), "pruned_fraction": round(pruned, 4), "rows_examined_per_coord": round(rows_read, 3),
            "cells_read_per_coord": round(cells_read, 3),
            "requests_per_step": requests, "requests_per_coord": round(requests / d, 3),
            "achieved_G_requests_per_s": round(ach, 1),
            "peak_G_requests_per_s": None if g_ms is None else round(d * r / (g_ms / 1e3) / 1e9, 1),
            "peak_probe": "gs_query_request_ceiling: the query's loads of all r rows, no median or store",
            "requests_frac_of_ceiling": None if g_ms is None else round(ach / (d * r / (g_ms / 1e3) / 1e9), 4),
            "time_vs_full_read_ceiling": None if g_ms is None else round(g_ms / q_ms, 4),
            "hbm": {"algorithmic_bytes": 4 * d, "achieved_GBps": round(4 * d / (q_ms / 1e3) / 1e9, 1),
                    "frac": round(4 * d / (q_ms / 1e3) / 1e9 / peaks["hbm_gbs"], 4)},
            "select_ms": None if ph["select"] is None else round(ph["select"], 4),
            "timed": "query and selection together (eager call)" if with_selection else
                     "query only (event nodes inside the step's graph)",
        }
    return k1, q


def probe_ceilings(run: Runner, reps: int = 3) -> dict:
    """The insert's and the query's measured request ceilings (medians of `reps`), run outside
    the timed region; the insert probe leaves the worker tables unspecified, and every step
    zeroes them first."""
    gs = run.gs
    out = {}
    if run.W >= 4 and (run.w.c & (run.w.c - 1)) == 0:
        import torch
        win = torch.empty(max(gs.gs_insert_request_ceiling_window_size(run.sk), 1 << 16), dtype=torch.uint8,
                          device=run.dev)
        out["insert_ms"] = statistics.median(gs.gs_insert_request_ceiling(run.sk, run.w.d, win, None, run.stream)
                                             for _ in range(reps))
        out["query_ms"] = statistics.median(gs.gs_query_request_ceiling(run.sk, run.w.d, win, None, run.stream)
                                            for _ in range(reps))
        del win
    return out


def measure(gs, w, variant, eager, steps, warmup, world, rank, dev, stream, peaks, peak_kind, sampler=None,
            want_e2e=False, probes=True, staged=False, group_width=0):
    """Time one workload; returns (summary dict, Runner still open for e2e)."""
    import torch
    want_host = want_e2e and variant == "error_feedback"
    run = Runner(gs, w, variant, eager, rank, dev, stream, steps + warmup, want_host, staged, group_width)
    flush = None
    streamed_bytes = w.P * w.d * 12
    if streamed_bytes < 2 * L2_BYTES:
        flush = torch.zeros(64 << 20, dtype=torch.float32, device=dev)   # 256 MB, twice the L2
    torch.cuda.synchronize()
    elapsed_ms, n_warm, n_by_plan = time_steps(run, steps, warmup, world, dev, sampler, flush)
    ph = run.phase_times(n_by_plan)
    pruned, rows_read, cells_read = run.query_rows() if variant != "heavymix" else (0.0, float(run.w.r),
                                                                                     float(run.w.r))
    pr = probe_ceilings(run) if probes else {}
    k1, q = rooflines(run, variant, ph, peaks, peak_kind, pr, pruned, rows_read, cells_read)
    value = whole_job_rate(world, w.P, w.d, steps, elapsed_ms / 1e3)
    res = {
        "value": value, "ms_per_step": round(elapsed_ms / steps, 4), "steps": steps, "warmup_steps_run": n_warm,
        "launch": "plan" if run.use_plan else "eager",
        "l2": ("flushed before every timed step (256 MB write, outside the step's events)" if flush is not None else
               f"inputs larger than L2 ({streamed_bytes / 1e9:.2f} GB of g,u,e streamed per step)"),
        "gpu_launches_per_step": launches_per_step(run, variant),
        "roofline": k1, "roofline_query": q,
        "insert_share_of_step": round(ph["insert"] / (elapsed_ms / steps), 3),
    }
    if run.streamed:
        res["streaming"] = {
            "worker_batch": run.batch,
            "gradient_generation_ms_per_step": None if ph["gen"] is None else round(ph["gen"], 3),
            "note": "every step draws fresh gradients for each batch of resident workers into one shared device "
                    "buffer set, then inserts the batch; generation is inside the step, outside the insert's events",
        }
        if ph["gen"] is not None:
            res["ms_per_step_without_generation"] = round(elapsed_ms / steps - ph["gen"], 4)
    if ph["query_select"] is not None:
        res["query_and_selection_ms"] = round(ph["query_select"], 4)
    del flush
    return res, run


def e2e_measure(gs, run: Runner, steps, warmup, world, dev):
    """End to end through the public API with host buffers: a host plan per gradient set (the
    uploads where needed, the step and the download of idx and vals are one graph), then a
    stream synchronisation so that the host can read the step's result."""
    import torch
    w = run.w
    P, d, k = w.P, w.d, w.k
    s = run.stream
    grad_dev = [torch.empty(d, dtype=torch.float32, device=dev) for _ in range(P)]
    idx_h = torch.empty(k, dtype=torch.int64).pin_memory()
    vals_h = torch.empty(k, dtype=torch.float32).pin_memory()
    hplans = []
    if run.use_plan:
        hplans = [gs.gs_step_host_plan_create(run.sk, run.us, run.es, hb, grad_dev, d, w.rho, k, idx_h, vals_h, run.ws)
                  for hb in run.host_pool]

    def host_step(t):
        if run.use_plan:
            gs.gs_plan_launch(hplans[t % len(hplans)], s)
            s.synchronize()
        else:
            gs.gs_step_host(run.sk, run.us, run.es, run.host_pool[t % len(run.host_pool)], grad_dev, d, w.rho, k,
                            idx_h, vals_h, run.ws, None, s)

    for t in range(max(warmup, len(hplans))):   # every plan once, at least W steps
        host_step(t)
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for t in range(steps):
        host_step(warmup + t)
    torch.cuda.synchronize()
    e2e_s = time.perf_counter() - t0
    barrier(world)
    e2e_s = dist_max(e2e_s, dev)
    for hp in hplans:
        gs.gs_plan_destroy(hp)
    return {"value": whole_job_rate(world, P, d, steps, e2e_s), "unit": UNIT, "h2d_bytes_per_step": P * d * 4,
            "d2h_bytes_per_step": k * (8 + 4), "ms_per_step": round(e2e_s * 1e3 / steps, 4),
            "call": "gs_step_host_plan_create + gs_plan_launch" if run.use_plan else "gs_step_host"}


def short_summary(res: dict, w) -> dict:
    k1, q = res["roofline"], res["roofline_query"]
    out = {
        "d": w.d, "P": w.P, "r": w.r, "c": w.c, "k": w.k, "steps": res["steps"], "launch": res["launch"],
        "value": res["value"], "unit": UNIT, "ms_per_step": res["ms_per_step"], "l2": res["l2"],
        "insert": {"avg_phase_ms": k1["avg_phase_ms"], "achieved": k1["achieved"], "frac": k1["frac"],
                   "row_passes": k1["row_passes"], "groups": k1["groups"],
                   "moved_bytes_per_worker_coord": k1["moved_bytes_per_worker_coord"],
                   "request_ceiling_ms": k1["co_bound"]["peak_ms"], "frac_of_request_ceiling": k1["co_bound"]["frac"],
                   "request_ceiling_frac_of_hbm": k1["co_bound"]["peak_frac_of_hbm"]},
        "query": None if q is None else {"avg_ms": q["avg_ms"], "pruned_fraction": q["pruned_fraction"],
                                          "rows_examined_per_coord": q["rows_examined_per_coord"],
                                          "cells_read_per_coord": q["cells_read_per_coord"],
                                          "achieved_G_requests_per_s": q["achieved_G_requests_per_s"],
                                          "peak_G_requests_per_s": q["peak_G_requests_per_s"],
                                          "requests_frac_of_ceiling": q["requests_frac_of_ceiling"],
                                          "time_vs_full_read_ceiling": q["time_vs_full_read_ceiling"],
                                          "select_ms": q["select_ms"], "timed": q["timed"]},
        "gpu_launches_per_step": res["gpu_launches_per_step"],
    }
    for key in ("streaming", "ms_per_step_without_generation", "query_and_selection_ms"):
        if key in res:
            out[key] = res[key]
    return out


def run_ours(args):
    import torch
    import paper_2108_06004_gb300 as gs

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    if not os.path.exists(gs.LIB_PATH):
        if rank == 0 or world == 1:
            from paper_2108_06004_gb300 import _build
            _build.build()
        barrier(world)
    gs.load_library()
    peaks, peak_kind = measured_peaks()
    stream = torch.cuda.current_stream()
    w = workloads.get_config(args.config)
    if args.d:
        w = shrink(w, args.d)
        args.profile_steps = True
    variant = args.variant
    quick = args.profile_steps

    sampler = None if quick else ClockSampler(gpu_uuid(dev))
    if sampler:
        sampler.start()
    staged = args.insert == "staged"
    if staged and (variant != "error_feedback" or (w.worker_batch and w.worker_batch < w.P)):
        raise SystemExit("--insert staged applies to the error_feedback step of a workload with all workers resident")
    res, run = measure(gs, w, variant, args.eager, args.steps, args.warmup, world, rank, dev, stream, peaks,
                       peak_kind, sampler, want_e2e=not (args.no_e2e or quick) and not staged,
                       probes=not quick, staged=staged, group_width=args.group_width)
    clocks = sampler.stop() if sampler else None

    e2e = None
    if not args.no_e2e and not quick and variant == "error_feedback" and not run.streamed and not staged:
        e2e = e2e_measure(gs, run, args.steps, args.warmup, world, dev)
    W, groups = run.W, run.groups
    run.close()
    del run
    torch.cuda.empty_cache()

    per_config = None
    if not args.no_per_config and not quick and variant == "error_feedback" and not staged:
        per_config = {}
        for name in sorted(workloads.CONFIGS, key=lambda n: workloads.CONFIGS[n].d):
            wc = workloads.get_config(name)
            if name == w.name:
                per_config[name] = short_summary(res, wc)
                continue
            steps = PER_CONFIG_STEPS.get(name, 5)
            rc, runc = measure(gs, wc, variant, args.eager, steps, max(3, min(args.warmup, 5)), world, rank, dev,
                               stream, peaks, peak_kind)
            per_config[name] = short_summary(rc, wc)
            runc.close()
            del runc
            torch.cuda.empty_cache()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not quick and variant == "error_feedback":
        cpu = cpu_baseline(w, steps=2)

    line = {
        "metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": w.name, "variant": variant, "launch": res["launch"], "insert": args.insert,
                   "warmup_steps_run": res["warmup_steps_run"], "d": w.d, "P": w.P, "r": w.r, "c": w.c, "k": w.k,
                   "rho": w.rho, "group_width": W, "groups": groups,
                   "parallelism": f"replicas{world}" if world > 1 else "single-gpu",
                   "l2": res["l2"], "d_steps_per_s": world * w.d * args.steps / (res["ms_per_step"] * args.steps / 1e3)},
        "roofline": res["roofline"], "roofline_query": res["roofline_query"], "cpu_baseline": cpu, "e2e": e2e,
        "gpu_launches": res["gpu_launches_per_step"] * args.steps, "clocks": clocks,
        "insert_share_of_step": res["insert_share_of_step"],
    }
    for key in ("streaming", "ms_per_step_without_generation", "query_and_selection_ms"):
        if key in res:
            line[key] = res[key]
    if per_config is not None:
        line["per_config"] = per_config
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# ---- the CPU oracle as baseline / reference arm -------------------------------------------

def _oracle_sample_step(w, t, d_s, k_s, coeffs, us, es):
    import oracle
    grads = workloads.make_gradients(w, t, range(w.P), d=d_s)
    t0 = time.perf_counter()
    res = oracle.step(us, es, grads, w.rho, coeffs, w.c, k_s)
    dt = time.perf_counter() - t0
    return dt, res


def host_cores() -> int:
    """Host cores this process may run on."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


def cpu_baseline(w, steps=1, d_s=CPU_SAMPLE_D):
    """The oracle, as it stands, on the first d_s coordinates of each worker's gradient
    (same P, r, c and rho; k scaled with d); the same unit as the metric."""
    import oracle
    d_s = min(d_s, w.d)
    k_s = max(1, round(w.k * d_s / w.d))
    coeffs = oracle.derive_coefficients(w.r, 20210813)
    us = [np.zeros(d_s, np.float32) for _ in range(w.P)]
    es = [np.zeros(d_s, np.float32) for _ in range(w.P)]
    total = 0.0
    for t in range(steps):
        dt, res = _oracle_sample_step(w, t, d_s, k_s, coeffs, us, es)
        total += dt
        us, es = res.us, res.es
    return {"value": w.P * d_s * steps / total, "unit": UNIT, "cores": 1, "cores_available": host_cores(),
            "processes": 1, "kind": "oracle",
            "sample": f"{steps} step(s) of the oracle on the first {d_s} coordinates of each of the {w.P} "
                      f"workers (r={w.r}, c={w.c}, k={k_s}), numpy single-threaded"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    import oracle
    w = workloads.get_config(args.config)
    per_step = REF_BUDGET_S / max(1, args.steps + args.warmup)
    d_s = 1 << 16
    while d_s * 2 <= min(w.d, 1 << 22) and 2 * d_s * w.P * ORACLE_S_PER_COORD <= per_step:
        d_s *= 2
    k_s = max(1, round(w.k * d_s / w.d))
    coeffs = oracle.derive_coefficients(w.r, 20210813)
    us = [np.zeros(d_s, np.float32) for _ in range(w.P)]
    es = [np.zeros(d_s, np.float32) for _ in range(w.P)]
    for t in range(args.warmup):
        _, res = _oracle_sample_step(w, t, d_s, k_s, coeffs, us, es)
        us, es = res.us, res.es
    total = 0.0
    for t in range(args.steps):
        dt, res = _oracle_sample_step(w, args.warmup + t, d_s, k_s, coeffs, us, es)
        total += dt
        us, es = res.us, res.es
    value = w.P * d_s * args.steps / total
    sample = (f"each step: the oracle on the first {d_s} coordinates of each of the {w.P} workers "
              f"(r={w.r}, c={w.c}, k={k_s}), numpy single-threaded")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(total * 1e3 / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "d": w.d, "P": w.P, "r": w.r, "c": w.c, "k": w.k, "rho": w.rho},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "cores_available": host_cores(), "processes": 1,
                         "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
